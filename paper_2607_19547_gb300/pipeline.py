"""One composition query (ChronoStitch Sec. 2, summary of the procedure) over the C ABI.

A query composes N stored chunk caches laid out as
    [text prefix P][chunk 0] ... [chunk N-1][text suffix S],   T tokens,
and runs the four calls of the hot path in stream order:
  1. cs_rebase_keys      all layers' keys, in place, local -> global coordinates (Eq. 3)
  2. cs_score_deviation  candidates = tokens of chunks 1..N-1 at the score layer (Eq. 5)
  3. cs_select_topk      k of them, written as the first k query positions
  4. cs_repair_attention the k selected rows plus the S suffix rows over the cache (Eq. 1)
Query tensors of the repaired rows and the fresh keys of the candidates come
from the model (projections and a shallow recompute, outside this library).
"""
from __future__ import annotations

import dataclasses

import torch

from . import cs_rebase_keys, cs_repair_attention, cs_score_deviation, cs_select_topk


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

    def step(self, k, v, q, k_fresh, pos_local, pos_global, stream=None):
        """Runs the four calls on `stream`; returns (attention output, query positions).

        k is re-based in place: after the call it is the composed cache."""
        s = self.shape
        cs_rebase_keys(k, pos_local, pos_global, theta=s.theta, sections=s.sections, stream=stream)
        cached = k[s.score_layer, s.cand0:s.cand0 + s.n_cand]
        cs_score_deviation(k_fresh, cached, out=self.score, stream=stream)
        cs_select_topk(self.score, s.k, s.cand0, out=self.qpos[:s.k], stream=stream)
        cs_repair_attention(q, k, v, self.qpos, out=self.out, stream=stream)
        return self.out, self.qpos


def compose_from_host(query: ComposedQuery, host: dict, dev: dict, out_host: dict, stream=None):
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
                             dev["pos_global"], stream=st)
        out_host["o"].copy_(o, non_blocking=True)
        out_host["qpos"].copy_(qpos, non_blocking=True)
    d2h = o.numel() * o.element_size() + qpos.numel() * qpos.element_size()
    return h2d, d2h
