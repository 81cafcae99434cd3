"""One composition query (ChronoStitch Sec. 2, summary of the procedure) over the C ABI.

A query composes N stored chunk caches laid out as
    [text prefix P][chunk 0] ... [chunk N-1][text suffix S],   T tokens,
and runs the four steps of the hot path in stream order:
  1. re-base             all layers' keys, in place, local -> global coordinates (Eq. 3)
  2. score               candidates = tokens of chunks 1..N-1 at the score layer (Eq. 5);
                         1 and 2 are one call, cs_rebase_and_score (one launch)
  3. cs_select_topk      k of them, written as the first k query positions
  4. cs_repair_attention the k selected rows plus the S suffix rows over the cache (Eq. 1)
Query tensors of the repaired rows and the fresh keys of the candidates come
from the model (projections and a shallow recompute, outside this library).

Options around the four calls:
  * policy: "3axis" (Eq. 3, the method), "scalar1d" (every token re-based to the
    scalar slot (i, i, i) of its sequence position, the 1-D re-index baseline of
    Sec. 2 / Table 1) or "naive" (stored keys used as they are, no re-base);
  * fresh_kv: the repaired rows' fresh keys and values [L, k, Hkv, D], written
    into the cache at the selected positions (cs_scatter_rows) before the
    attention, as the recompute does layer by layer (Sec. 2);
  * shallow_recompute(): the attention part of the shallow recompute, every
    candidate as a query row over the first layers (the 2 c_a |C| T term of
    Eq. 6), run with the same attention kernel;
  * GraphedQuery: a whole end-to-end query (input copies, the launches, output
    copies) captured once as a CUDA graph and replayed with one launch;
  * PipelinedQuery: the same with uploads, kernels and downloads overlapped layer
    group by layer group on three streams (short first and last groups), also one graph;
  * QueryStream: a stream of queries with several in flight (per slot, captured graphs of
    the uploads, the launches and the downloads on shared upload, compute and download
    streams), so one query's uploads and another's downloads overlap the computation
    between them.
"""
from __future__ import annotations

import dataclasses

import torch

from . import (cs_rebase_and_score, cs_rebase_keys, cs_repair_attention, cs_scatter_rows,
               cs_score_deviation, cs_select_topk)

POLICIES = ("3axis", "scalar1d", "naive")


@dataclasses.dataclass
class QueryShape:
    n_layers: int
    T: int
    hq: int
    hkv: int
    cand0: int          # global index of the first candidate token
    n_cand: int         # candidates (later-chunk visual tokens)
    k: int              # tokens to repair
    suffix: int         # text suffix rows that also query the cache (the last S tokens)
    score_layer: int = 1
    head_dim: int = 128
    theta: float = 1e6
    sections: tuple = (16, 24, 24)

    @property
    def M(self) -> int:
        return self.k + self.suffix


class ComposedQuery:
    """Device scratch for one query shape: scores, query positions and the output."""

    def __init__(self, shape: QueryShape, dtype: torch.dtype, device="cuda"):
        self.shape = shape
        s = shape
        self.score = torch.empty(s.n_cand, dtype=torch.float32, device=device)
        self.qpos = torch.empty(s.M, dtype=torch.int32, device=device)
        if s.suffix:
            self.qpos[s.k:] = torch.arange(s.T - s.suffix, s.T, dtype=torch.int32, device=device)
        self.out = torch.empty((s.n_layers, s.M, s.hq, s.head_dim), dtype=dtype, device=device)
        self.device = device
        self._scalar_targets = None
        self._cand_pos = None

    def scalar_targets(self) -> torch.Tensor:
        """int32 [T, 3] with row i = (i, i, i): the scalar re-index targets."""
        if self._scalar_targets is None:
            i = torch.arange(self.shape.T, dtype=torch.int32, device=self.device)
            self._scalar_targets = torch.stack([i, i, i], dim=1).contiguous()
        return self._scalar_targets

    def step(self, k, v, q, k_fresh, pos_local, pos_global, stream=None, policy="3axis",
             fresh_kv=None):
        """Runs the four calls on `stream`; returns (attention output, query positions).

        k is re-based in place: after the call it is the composed cache (with the
        repaired rows' fresh keys and values when fresh_kv is given)."""
        s = self.shape
        if policy not in POLICIES:
            raise ValueError(f"policy must be one of {POLICIES}")
        if policy == "naive":
            cached = k[s.score_layer, s.cand0:s.cand0 + s.n_cand]
            cs_score_deviation(k_fresh, cached, out=self.score, stream=stream)
        else:   # re-base and score in one launch (the score reads the rows just re-based)
            target = pos_global if policy == "3axis" else self.scalar_targets()
            cs_rebase_and_score(k, pos_local, target, k_fresh, s.score_layer, s.cand0,
                                score_out=self.score, theta=s.theta, sections=s.sections,
                                stream=stream)
        cs_select_topk(self.score, s.k, s.cand0, out=self.qpos[:s.k], stream=stream)
        if fresh_kv is not None:
            k_rows, v_rows = fresh_kv
            cs_scatter_rows(k, k_rows, self.qpos[:s.k], stream=stream)
            cs_scatter_rows(v, v_rows, self.qpos[:s.k], stream=stream)
        cs_repair_attention(q, k, v, self.qpos, out=self.out, stream=stream)
        return self.out, self.qpos

    def shallow_recompute(self, q_cand, k, v, stream=None, out=None):
        """Attention of every candidate token over the composed cache for the first
        q_cand.shape[0] layers (q_cand [layers, n_cand, Hq, D]); returns [layers, n_cand, Hq, D]."""
        s = self.shape
        if self._cand_pos is None:
            self._cand_pos = torch.arange(s.cand0, s.cand0 + s.n_cand, dtype=torch.int32,
                                          device=self.device)
        nl = q_cand.shape[0]
        return cs_repair_attention(q_cand, k[:nl], v[:nl], self._cand_pos, out=out, stream=stream)


class GraphedQuery:
    """One whole end-to-end query captured as a CUDA graph for fixed buffers: the host->device
    copies of k, v, q and k_fresh, the three launches of the step, and the device->host copies
    of the output and the query positions.  replay() runs all of it with one graph launch, on
    the current contents of the host buffers.

    host / dev / out_host as for compose_from_host.  The first step runs eagerly (it also
    performs the library's one-time set-up) before the capture."""

    def __init__(self, query: ComposedQuery, host: dict, dev: dict, out_host: dict,
                 policy="3axis"):
        self.query, self.host, self.dev, self.out_host = query, host, dev, out_host
        self.policy = policy
        side = torch.cuda.Stream(device=dev["k"].device)
        side.wait_stream(torch.cuda.current_stream(dev["k"].device))
        with torch.cuda.stream(side):
            self.h2d, self.d2h = compose_from_host(query, host, dev, out_host, stream=side,
                                                   policy=policy)
        side.synchronize()
        self.graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(self.graph, stream=side):
            compose_from_host(query, host, dev, out_host, stream=side, policy=policy)

    def replay(self):
        """Runs the captured query on the current stream's device (asynchronously)."""
        self.graph.replay()
        return self.h2d, self.d2h


def _group_launches(q: ComposedQuery, dev: dict, a: int, b: int, policy: str, stream):
    """The launches of one query for layers [a, b) on `stream`: re-base (for the group that
    holds the score layer, with the score and the selection), then the repair attention of
    those layers.  Every group's attention reads the selection, which the score layer's group
    makes, so that group comes first in stream order."""
    s = q.shape
    k = dev["k"][a:b]
    target = dev["pos_global"] if policy == "3axis" else q.scalar_targets()
    if a <= s.score_layer < b:
        if policy == "naive":
            cached = dev["k"][s.score_layer, s.cand0:s.cand0 + s.n_cand]
            cs_score_deviation(dev["k_fresh"], cached, out=q.score, stream=stream)
        else:
            cs_rebase_and_score(k, dev["pos_local"], target, dev["k_fresh"], s.score_layer - a,
                                s.cand0, score_out=q.score, theta=s.theta, sections=s.sections,
                                stream=stream)
        cs_select_topk(q.score, s.k, s.cand0, out=q.qpos[:s.k], stream=stream)
    elif policy != "naive":
        cs_rebase_keys(k, dev["pos_local"], target, theta=s.theta, sections=s.sections,
                       stream=stream)
    cs_repair_attention(dev["q"][a:b], k, dev["v"][a:b], q.qpos, out=q.out[a:b], stream=stream)


def plan_layer_groups(n_layers: int, score_layer: int, group_layers: int = 4, bounds=None):
    """Layer groups of a pipelined query, as (first, end) pairs covering [0, n_layers).

    By default: a short first group that reaches the score layer (the pipeline waits for its
    upload, so the selection runs as early as possible), groups of group_layers, and a short
    last group of 2 layers (its compute and download trail the last upload).  bounds, when
    given, are the group boundaries themselves: they must rise strictly from 0 to n_layers,
    and the first group must hold the score layer (every group's attention reads the
    selection that the score layer's group makes)."""
    if n_layers < 1:
        raise ValueError("n_layers must be at least 1")
    if not 0 <= score_layer < n_layers:
        raise ValueError("score_layer must be a layer of the cache")
    if bounds is None:
        if group_layers < 1:
            raise ValueError("group_layers must be at least 1")
        L = n_layers
        lead, tail = min(L, max(2, score_layer + 1)), 2
        bounds = [0, lead]
        while bounds[-1] + group_layers < L - tail:
            bounds.append(bounds[-1] + group_layers)
        if L - tail > bounds[-1]:
            bounds.append(L - tail)
        if L > bounds[-1]:
            bounds.append(L)
    bounds = [int(x) for x in bounds]
    if (len(bounds) < 2 or bounds[0] != 0 or bounds[-1] != n_layers
            or any(b <= a for a, b in zip(bounds[:-1], bounds[1:]))):
        raise ValueError("bounds must rise strictly from 0 to n_layers")
    if not score_layer < bounds[1]:
        # every group's attention reads the selection, which the score layer's group makes
        raise ValueError("the first group must hold the score layer")
    return list(zip(bounds[:-1], bounds[1:]))


class PipelinedQuery:
    """An end-to-end query from host buffers with the copies and the kernels overlapped layer
    group by layer group, captured as one CUDA graph.

    Three streams: uploads (K, V and Q of one group of layers, the fresh keys first), compute
    (the group's re-base; for the group holding the score layer also its score and the
    selection; then the group's attention), downloads (the group's output, and the query
    positions at the end).  Each group's compute waits for its uploads and each download for
    its compute, so group g+1 uploads while group g computes and group g-1 downloads.  The
    kernels are the same calls as ComposedQuery.step on layer slices (every call takes a
    layer count and stride), so the result is identical.  replay() runs it all with one graph
    launch on the current contents of the host buffers."""

    def __init__(self, query: ComposedQuery, host: dict, dev: dict, out_host: dict,
                 group_layers: int = 4, policy: str = "3axis", bounds=None):
        if policy not in POLICIES:
            raise ValueError(f"policy must be one of {POLICIES}")
        s = query.shape
        self.query, self.host, self.dev, self.out_host = query, host, dev, out_host
        self.groups = plan_layer_groups(s.n_layers, s.score_layer, group_layers, bounds)
        device = dev["k"].device
        self.s_in, self.s_c, self.s_out = (torch.cuda.Stream(device=device) for _ in range(3))
        self.h2d = sum(host[n].numel() * host[n].element_size() for n in ("k", "v", "q", "k_fresh"))
        self.d2h = query.out.numel() * query.out.element_size() + query.qpos.numel() * 4
        self.s_c.wait_stream(torch.cuda.current_stream(device))
        with torch.cuda.stream(self.s_c):
            self._record(policy)          # eager run: one-time set-up of the library
        self.s_c.synchronize()
        self.graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(self.graph, stream=self.s_c):
            self._record(policy)

    def _record(self, policy):
        q, s, host, dev, out_host = self.query, self.query.shape, self.host, self.dev, self.out_host
        s_in, s_c, s_out = self.s_in, self.s_c, self.s_out
        s_in.wait_stream(s_c)
        s_out.wait_stream(s_c)
        with torch.cuda.stream(s_in):
            dev["k_fresh"].copy_(host["k_fresh"], non_blocking=True)
        for a, b in self.groups:
            with torch.cuda.stream(s_in):
                for n in ("k", "v", "q"):
                    dev[n][a:b].copy_(host[n][a:b], non_blocking=True)
            s_c.wait_stream(s_in)
            with torch.cuda.stream(s_c):
                _group_launches(q, dev, a, b, policy, s_c)
            s_out.wait_stream(s_c)
            with torch.cuda.stream(s_out):
                out_host["o"][a:b].copy_(q.out[a:b], non_blocking=True)
        with torch.cuda.stream(s_out):
            out_host["qpos"].copy_(q.qpos, non_blocking=True)
        s_c.wait_stream(s_in)
        s_c.wait_stream(s_out)

    def replay(self):
        """Runs the captured query (asynchronously, ordered after the current stream's work)."""
        self.graph.replay()
        return self.h2d, self.d2h


class QueryStream:
    """A stream of end-to-end queries from host memory, n_slots of them in flight.

    Each slot owns its device buffers (keys, values, queries and fresh keys; scores, query
    positions and output through its own ComposedQuery), pinned host output buffers, and, for
    each of a query's layer parts (a short first part that holds the score layer, the middle,
    a short last part), captured CUDA graphs of the part's uploads, launches and downloads.
    Query i runs in slot i % n_slots: its uploads go on the shared upload stream once the
    slot's previous query has finished computing (its buffers are then free), each part's
    launches on the shared compute stream after that part's uploads (and after the slot's
    previous download of the same part, which reads the output buffer), each part's download on
    the shared download stream after its launches.  The queries' computations thus run one
    after another while later queries upload and earlier ones download: in steady state a query
    costs the longest of its upload, compute and download times, and the parts shorten what the
    first query waits for its inputs and the last one for its output.  Every query copies its
    own inputs in and its result out.

    host: the pinned host inputs (k, v, q, k_fresh), one dict shared by every slot or a list
    with one dict per slot; pos_local, pos_global: device coordinates, shared read-only."""

    def __init__(self, shape: QueryShape, dtype: torch.dtype, host, pos_local, pos_global,
                 n_slots: int = 2, policy: str = "3axis"):
        if n_slots < 1:
            raise ValueError("n_slots must be at least 1")
        if policy not in POLICIES:
            raise ValueError(f"policy must be one of {POLICIES}")
        hosts = list(host) if isinstance(host, (list, tuple)) else [host] * n_slots
        if len(hosts) != n_slots:
            raise ValueError("host must be one dict or one dict per slot")
        self.device = pos_local.device
        self.n_slots = n_slots
        self.parts = plan_layer_groups(shape.n_layers, shape.score_layer,
                                       group_layers=shape.n_layers)
        self.s_up, self.s_c, self.s_down = (torch.cuda.Stream(device=self.device) for _ in range(3))
        names = ("k", "v", "q", "k_fresh")
        self.h2d = sum(hosts[0][n].numel() * hosts[0][n].element_size() for n in names)
        self.slots = []
        side = torch.cuda.Stream(device=self.device)
        side.wait_stream(torch.cuda.current_stream(self.device))
        last = len(self.parts) - 1
        for h in hosts:
            q = ComposedQuery(shape, dtype, device=self.device)
            dev = {n: torch.empty(h[n].shape, dtype=h[n].dtype, device=self.device) for n in names}
            dev.update(pos_local=pos_local, pos_global=pos_global)
            out_host = {"o": torch.empty(q.out.shape, dtype=q.out.dtype).pin_memory(),
                        "qpos": torch.empty(shape.M, dtype=torch.int32).pin_memory()}

            def upload(p, a, b, h=h, dev=dev):
                if p == 0:
                    dev["k_fresh"].copy_(h["k_fresh"], non_blocking=True)
                for n in ("k", "v", "q"):
                    dev[n][a:b].copy_(h[n][a:b], non_blocking=True)

            def compute(p, a, b, q=q, dev=dev):
                _group_launches(q, dev, a, b, policy, torch.cuda.current_stream(self.device))

            def download(p, a, b, q=q, out_host=out_host):
                out_host["o"][a:b].copy_(q.out[a:b], non_blocking=True)
                if p == last:
                    out_host["qpos"].copy_(q.qpos, non_blocking=True)

            phases = (upload, compute, download)
            with torch.cuda.stream(side):          # eager run: the library's one-time set-up
                for p, (a, b) in enumerate(self.parts):
                    for fn in phases:
                        fn(p, a, b)
            side.synchronize()
            graphs = []
            for p, (a, b) in enumerate(self.parts):
                per_part = []
                for fn in phases:
                    g = torch.cuda.CUDAGraph()
                    with torch.cuda.graph(g, stream=side):
                        fn(p, a, b)
                    per_part.append(g)
                graphs.append(per_part)
            self.slots.append({"query": q, "dev": dev, "out_host": out_host, "graphs": graphs,
                               "ev": [[torch.cuda.Event() for _ in range(3)] for _ in self.parts],
                               "used": False})
        q0 = self.slots[0]["query"]
        self.d2h = q0.out.numel() * q0.out.element_size() + q0.qpos.numel() * 4

    def out_host(self, slot: int) -> dict:
        """The pinned host outputs (o, qpos) of `slot`: its last query's result."""
        return self.slots[slot]["out_host"]

    def run(self, n_queries: int):
        """Launches n_queries queries, query i in slot i % n_slots, ordered after the current
        stream's work; the current stream then waits for all of them (asynchronous to the
        host).  Returns the bytes copied per query (host->device, device->host)."""
        cur = torch.cuda.current_stream(self.device)
        for st in (self.s_up, self.s_c, self.s_down):
            st.wait_stream(cur)
        last = len(self.parts) - 1
        for i in range(n_queries):
            s = self.slots[i % self.n_slots]
            if s["used"]:
                # the slot's previous query has read its inputs once its last part is computed
                self.s_up.wait_event(s["ev"][last][1])
            for p in range(len(self.parts)):
                with torch.cuda.stream(self.s_up):
                    s["graphs"][p][0].replay()
                    s["ev"][p][0].record(self.s_up)
            for p in range(len(self.parts)):
                ev_up, ev_c, ev_down = s["ev"][p]
                self.s_c.wait_event(ev_up)
                if s["used"]:
                    self.s_c.wait_event(ev_down)    # this part's previous output is downloaded
                with torch.cuda.stream(self.s_c):
                    s["graphs"][p][1].replay()
                    ev_c.record(self.s_c)
                self.s_down.wait_event(ev_c)
                with torch.cuda.stream(self.s_down):
                    s["graphs"][p][2].replay()
                    ev_down.record(self.s_down)
            s["used"] = True
        for st in (self.s_up, self.s_c, self.s_down):
            cur.wait_stream(st)
        return self.h2d, self.d2h


def compose_from_host(query: ComposedQuery, host: dict, dev: dict, out_host: dict, stream=None,
                      policy="3axis"):
    """End-to-end query from host memory: copies the step's inputs in, runs it, copies the result out.

    host / dev: dicts with k, v, q, k_fresh (pinned host tensors / device tensors of the
    same shapes); coordinates are expected to be device-resident already in dev.
    out_host: pinned host tensors "o" and "qpos" that receive the result.
    Returns the number of bytes copied (host->device, device->host)."""
    st = torch.cuda.current_stream() if stream is None else stream
    h2d = 0
    with torch.cuda.stream(st):
        for name in ("k", "v", "q", "k_fresh"):
            dev[name].copy_(host[name], non_blocking=True)
            h2d += host[name].numel() * host[name].element_size()
        o, qpos = query.step(dev["k"], dev["v"], dev["q"], dev["k_fresh"], dev["pos_local"],
                             dev["pos_global"], stream=st, policy=policy)
        out_host["o"].copy_(o, non_blocking=True)
        out_host["qpos"].copy_(qpos, non_blocking=True)
    d2h = o.numel() * o.element_size() + qpos.numel() * qpos.element_size()
    return h2d, d2h
