"""One pass of Conduit's hot path over a batch: the user-facing step.

``RefreshPipeline.step()`` enqueues, on one CUDA stream and through the C ABI:
  1. conduit_score        scoring pass over the reused visual cache (Eqs. 6-8)
  2. conduit_select_topk  amplification + one global top-k per request (Eqs. 9-11)
     (steps 1 and 2 as one call, conduit_score_select_topk, which runs the
     scoring tail and the selection as one launch)
  3. conduit_kv_exchange  stale K/V rows of the selected tokens out, fresh rows in
                          (conduit_kv_gather + conduit_kv_scatter in one launch)
  4. conduit_refresh_attn causal attention of the refreshed rows over the patched cache
``selection="quota"`` replaces step 2 by conduit_select_quota (explicit
per-image quotas, App. D.3). Scoring variants (conduit_score_ex): ``statistic="rms"`` (Eq. 4),
``value_norm="none"`` (attention alone) and ``extra_lse`` (full-context
softmax). With ``value_norm="side_cache"`` the pipeline keeps the value-norm
side cache (Sec. 4.3, App. C.2): it is built once at construction
(conduit_value_norms), step 1 reads it instead of V, and step 3 is followed by
conduit_value_norms_update for the rewritten rows, so every step's scores are
bitwise those of the pass that reads V.
All buffers are allocated once at construction, so a step allocates nothing
and can be captured in a CUDA graph (``capture()``). ``step_from_host()`` is
the end-to-end form: it copies the step's inputs from pinned host memory,
runs the step, and copies the selection and the refresh output back;
``DoubleBuffered`` alternates two pipelines so that one step's copies overlap
the previous step's kernels.
"""

from __future__ import annotations

from typing import Optional, Sequence

import torch

from . import conduit as C


class RefreshPipeline:
    def __init__(self, k: torch.Tensor, v: torch.Tensor, q: torch.Tensor, num_q_heads: int,
                 tok_off, img_off, req_img_off, q_off, ratios: Sequence[float],
                 fresh: dict, lam: float = 1.0, layers: Optional[Sequence[int]] = None,
                 page_size: int = 0, page_table: Optional[torch.Tensor] = None,
                 budgets: Optional[Sequence[int]] = None, statistic: str = "mean",
                 value_norm: str = "v", extra_lse: Optional[torch.Tensor] = None,
                 selection: str = "global"):
        dev = k.device
        self.device = dev
        self.kv = C.KvCache(k, v, num_q_heads, page_size, page_table)
        self._page_size = page_size
        self.batch = C.Batch(tok_off, img_off, req_img_off, q_off, device=dev)
        self.q = q
        self.lam = float(lam)
        self.layers = None if layers is None else list(layers)
        tok = self.batch.tok_off.tolist()
        n_r = [tok[r + 1] - tok[r] for r in range(self.batch.num_requests)]
        if budgets is None:
            budgets = [C.conduit_budget(r, n) for r, n in zip(ratios, n_r)]
        self.budgets = [int(x) for x in budgets]
        self.idx_off, self.idx_off_dev = C.idx_offsets(self.budgets, dev)
        self.n_sel = int(self.idx_off[-1])
        n_tot, K = self.batch.n_tot, self.batch.num_images
        f32 = dict(dtype=torch.float32, device=dev)
        self.s = torch.empty(n_tot, **f32)
        self.attn_sum = torch.empty(n_tot, **f32)
        self.g = torch.empty(K, **f32)
        self.s_hat = torch.empty(n_tot, **f32)
        self.coeff = torch.empty(K, **f32)
        self.mask = torch.empty(n_tot, dtype=torch.uint8, device=dev)
        self.idx = torch.empty(max(self.n_sel, 1), dtype=torch.int32, device=dev)
        self.status = torch.zeros(1, dtype=torch.int32, device=dev)
        nl = 0 if self.layers is None else len(self.layers)
        self.statistic, self.value_norm, self.extra_lse = statistic, value_norm, extra_lse
        self.vnorm = C.conduit_value_norms(self.kv, self.batch) if value_norm == "side_cache" else None
        self.plain = statistic == "mean" and value_norm == "v" and extra_lse is None
        opts = C.score_opts(statistic, value_norm, self.vnorm, extra_lse)
        if selection not in ("global", "quota"):
            raise ValueError("selection must be 'global' or 'quota'")
        # the fused call's workspace starts with the scoring call's, so one
        # buffer serves conduit_score(_ex) and conduit_score_select_topk
        ws_bytes = (C.conduit_score_select_topk_workspace_size if selection == "global"
                    else C.conduit_score_ex_workspace_size)(self.kv, self.batch, nl, opts)
        self.ws_score = torch.empty(max(ws_bytes, 1), dtype=torch.uint8, device=dev)
        self.selection = selection
        self.quota = torch.empty(K, dtype=torch.int32, device=dev) if selection == "quota" else None
        sel_ws = (C.conduit_select_quota_workspace_size if selection == "quota"
                  else C.conduit_select_workspace_size)(self.batch)
        self.ws_sel = torch.empty(max(sel_ws, 1), dtype=torch.uint8, device=dev)
        need = C.conduit_refresh_workspace_size(self.kv, self.batch, self.idx_off)
        self.ws_ref = torch.empty(need, dtype=torch.uint8, device=dev) if need else None
        L, Hkv, Hq, d = self.kv.num_layers, self.kv.num_kv_heads, num_q_heads, self.kv.head_dim
        self.q_rows = fresh["q_rows"]
        self.k_rows = fresh["k_rows"]
        self.v_rows = fresh["v_rows"]
        assert self.q_rows.shape == (L, self.n_sel, Hq, d)
        self.k_old = torch.empty((L, self.n_sel, Hkv, d), dtype=k.dtype, device=dev)
        self.v_old = torch.empty_like(self.k_old)
        self.out = torch.empty_like(self.q_rows)
        self.graph = None
        self._copy = None  # copy stream and events of step_from_host
        self._out_graph = None  # refresh with the output copied out per layer chunk (step_from_host)

    # ----------------------------------------------------------------- steps
    def score(self, stream=None):
        if self.plain:
            C.conduit_score(self.kv, self.batch, self.q, self.layers, self.s, self.attn_sum, self.g,
                            self.ws_score, self.status, stream)
        else:
            C.conduit_score_ex(self.kv, self.batch, self.q, self.layers, self.statistic,
                               self.value_norm, self.vnorm, self.extra_lse, self.s, self.attn_sum,
                               self.g, self.ws_score, self.status, stream)

    def select(self, stream=None):
        if self.selection == "quota":
            C.conduit_select_quota(self.batch, self.s, self.g, self.lam, self.idx_off, self.idx_off_dev,
                                   self.idx, self.mask, self.s_hat, self.coeff, self.quota, self.ws_sel,
                                   self.status, stream)
        else:
            C.conduit_select_topk(self.batch, self.s, self.g, self.lam, self.idx_off, self.idx_off_dev,
                                  self.idx, self.mask, self.s_hat, self.coeff, self.ws_sel,
                                  self.status, stream)

    def exchange(self, stream=None):
        C.conduit_kv_exchange(self.kv, self.batch, self.idx, self.idx_off, self.idx_off_dev,
                              self.k_old, self.v_old, self.k_rows, self.v_rows, stream)

    def norm_update(self, stream=None):
        if self.vnorm is not None:
            C.conduit_value_norms_update(self.kv, self.batch, self.idx, self.idx_off, self.idx_off_dev,
                                         self.vnorm, stream)

    def refresh_attn(self, stream=None):
        C.conduit_refresh_attn(self.kv, self.batch, self.idx, self.idx_off, self.idx_off_dev,
                               self.q_rows, self.out, self.ws_ref, self.status, stream)

    def score_select(self, stream=None):
        """Steps 1 and 2. With the global rule, one call (conduit_score_select_topk):
        the same results as score() then select(), in fewer launches."""
        if self.selection == "quota":
            self.score(stream)
            self.select(stream)
            return
        C.conduit_score_select_topk(self.kv, self.batch, self.q, self.lam, self.idx_off, self.idx_off_dev,
                                    self.layers, self.statistic, self.value_norm, self.vnorm, self.extra_lse,
                                    self.s, self.attn_sum, self.g, self.idx, self.mask, self.s_hat,
                                    self.coeff, self.ws_score, self.status, stream)

    def refresh(self, stream=None):
        self.exchange(stream)
        self.norm_update(stream)
        self.refresh_attn(stream)

    def _score_select_step(self):
        if self.graph is not None:
            self.graph[0].replay()
        else:
            self.score_select()

    def _refresh_step(self):
        if self.graph is not None:
            self.graph[1].replay()
        else:
            self.refresh()

    def step(self, stream=None):
        """One pass of the whole hot path (launches only; asynchronous)."""
        if self.graph is not None:
            self.graph[2].replay()
            return
        self.score_select(stream)
        self.refresh(stream)

    def capture(self):
        """Capture the step as CUDA graphs: scoring and selection, exchange and
        refresh (step_from_host starts the first while the second's inputs are
        still arriving), and the whole step in one graph, which later step()
        calls replay (one graph launch per step)."""
        s = torch.cuda.Stream(device=self.device)
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            self.score_select(s)
            self.refresh(s)
        torch.cuda.current_stream().wait_stream(s)
        torch.cuda.synchronize()
        g1, g2, g3 = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
        with torch.cuda.graph(g1):
            self.score_select()
        with torch.cuda.graph(g2):
            self.refresh()
        with torch.cuda.graph(g3):
            self.score_select()
            self.refresh()
        self.graph = (g1, g2, g3)

    # ------------------------------------------------------------- end to end
    def host_buffers(self) -> dict:
        """Pinned host copies of everything a step consumes and returns."""
        pin = lambda t: torch.empty(t.shape, dtype=t.dtype, pin_memory=True).copy_(t)
        return {
            "k": pin(self.kv.k), "v": pin(self.kv.v), "q": pin(self.q),
            "q_rows": pin(self.q_rows), "k_rows": pin(self.k_rows), "v_rows": pin(self.v_rows),
            "idx": torch.empty(self.idx.shape, dtype=torch.int32, pin_memory=True),
            "out": torch.empty(self.out.shape, dtype=self.out.dtype, pin_memory=True),
        }

    def step_from_host(self, host: dict, after: Optional[torch.cuda.Event] = None):
        """H2D copy of the cache, queries and fresh rows; the step; D2H of idx and out.

        The copies run on a stream of their own: the scoring pass starts once
        the cache and the queries have arrived, while the fresh rows (needed
        only by the exchange and the refresh) are still being copied; the
        refresh runs in layer chunks, each chunk's output copied back while
        the next chunks compute. The copies wait for everything enqueued on
        the current stream before the call, or, given ``after``, for that
        event only (the caller vouches that this pipeline's buffers are free
        once it has fired; see ``DoubleBuffered``).
        """
        cs = torch.cuda.current_stream(self.device)
        if self._copy is None:
            self._copy = (torch.cuda.Stream(device=self.device), torch.cuda.Event(), torch.cuda.Event())
        xs, ev_in, ev_fresh = self._copy
        if after is None:
            xs.wait_stream(cs)  # the device buffers are free once the previous step is done
        else:
            xs.wait_event(after)
        with torch.cuda.stream(xs):
            for name, dst in (("k", self.kv.k), ("v", self.kv.v), ("q", self.q)):
                dst.copy_(host[name], non_blocking=True)
            ev_in.record(xs)
            for name, dst in (("q_rows", self.q_rows), ("k_rows", self.k_rows), ("v_rows", self.v_rows)):
                dst.copy_(host[name], non_blocking=True)
            ev_fresh.record(xs)
        cs.wait_event(ev_in)
        self._score_select_step()
        host["idx"].copy_(self.idx, non_blocking=True)
        cs.wait_event(ev_fresh)
        self._refresh_to_host(host["out"])

    def _refresh_chunks(self, host_out, side):
        """Exchange, then the refresh attention layer chunk by layer chunk, each
        chunk's output copied to host_out on `side` while later chunks run."""
        cs = torch.cuda.current_stream(self.device)
        self.exchange()
        self.norm_update()
        for view, (l0, l1) in self._chunk_views:
            C.conduit_refresh_attn(view, self.batch, self.idx, self.idx_off, self.idx_off_dev,
                                   self.q_rows[l0:l1], self.out[l0:l1], self.ws_ref, self.status)
            side.wait_stream(cs)
            with torch.cuda.stream(side):
                host_out[l0:l1].copy_(self.out[l0:l1], non_blocking=True)
        cs.wait_stream(side)

    def _refresh_to_host(self, host_out, chunks: int = 4):
        if self._out_graph is None or self._out_graph[1] is not host_out:
            L = self.kv.num_layers
            bounds = sorted({round(i * L / chunks) for i in range(chunks + 1)})
            kv = self.kv
            self._chunk_views = [
                (C.KvCache(kv.k[l0:l1], kv.v[l0:l1], kv.num_q_heads, self._page_size, kv.page_table),
                 (l0, l1))
                for l0, l1 in zip(bounds[:-1], bounds[1:])]
            side = torch.cuda.Stream(device=self.device)
            if self.graph is None:
                self._out_graph = (None, host_out, side)
            else:
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g):
                    self._refresh_chunks(host_out, side)
                self._out_graph = (g, host_out, side)
        g, _, side = self._out_graph
        if g is not None:
            g.replay()
        else:
            self._refresh_chunks(host_out, side)

    def h2d_bytes(self) -> int:
        ts = (self.kv.k, self.kv.v, self.q, self.q_rows, self.k_rows, self.v_rows)
        return sum(t.numel() * t.element_size() for t in ts)

    def d2h_bytes(self) -> int:
        return self.idx.numel() * 4 + self.out.numel() * self.out.element_size()


class DoubleBuffered:
    """Two pipelines of one batch shape, stepped alternately from host buffers.

    A step's host-to-device copies wait only for the previous step on the
    same pipeline, so they run while the other pipeline's step computes, and
    back-to-back steps are bound by the host link instead of by copies and
    kernels in series. Both pipelines' kernels run on the current stream, in
    call order, and each step's device-to-host copies complete before the
    next step's kernels start.
    """

    def __init__(self, first: RefreshPipeline, second: RefreshPipeline):
        if first.kv.k.shape != second.kv.k.shape or first.budgets != second.budgets:
            raise ValueError("DoubleBuffered needs two pipelines of the same batch shape")
        # a pipeline keeps the tensors it was built on; the copies of one step
        # would overwrite what the other pipeline's step is reading
        bufs = lambda p: {t.data_ptr() for t in (p.kv.k, p.kv.v, p.q, p.q_rows, p.k_rows, p.v_rows)}
        if bufs(first) & bufs(second):
            raise ValueError("DoubleBuffered needs two pipelines over separate device buffers")
        self.pipes = (first, second)
        self._done = [None, None]
        self._next = 0

    def start_after(self, event: torch.cuda.Event):
        """Order the next copies of both pipelines after ``event`` (and after
        every earlier step, which it must follow)."""
        self._done = [event, event]

    def step_from_host(self, host: dict) -> RefreshPipeline:
        """One step on the next pipeline; returns the pipeline that ran it."""
        i = self._next
        p = self.pipes[i]
        p.step_from_host(host, after=self._done[i])
        ev = torch.cuda.Event()
        ev.record(torch.cuda.current_stream(p.device))
        self._done[i] = ev
        self._next = i ^ 1
        return p


def from_inputs(inputs: dict, lam: float = 1.0, paged: Optional[bool] = None,
                layers=None, budgets=None, fresh: Optional[dict] = None,
                **score_variant) -> RefreshPipeline:
    """A pipeline over a batch drawn by ``synth.make_inputs``."""
    from . import synth
    w = inputs["workload"]
    dev = inputs["k"].device
    tok = inputs["tok_off"].tolist()
    n_r = [tok[r + 1] - tok[r] for r in range(len(tok) - 1)]
    if budgets is None:
        budgets = [C.conduit_budget(r, n) for r, n in zip(inputs["ratios"], n_r)]
    if fresh is None:
        fresh = synth.make_fresh_rows(w, sum(budgets), device=dev)
    paged = bool(w.page_size) if paged is None else paged
    k, v, table, ps = inputs["k"], inputs["v"], None, 0
    if paged:
        ps = w.page_size or 16
        k, table = synth.to_paged(inputs["k"], tok, ps, w.seed)
        v, _ = synth.to_paged(inputs["v"], tok, ps, w.seed)
    return RefreshPipeline(k, v, inputs["q"], w.num_q_heads, inputs["tok_off"], inputs["img_off"],
                           inputs["req_img_off"], inputs["q_off"], inputs["ratios"], fresh, lam=lam,
                           layers=layers, page_size=ps, page_table=table, budgets=budgets,
                           **score_variant)
