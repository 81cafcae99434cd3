"""GraphedQuery: one end-to-end query (input copies, the launches, output copies) captured as
a CUDA graph.  Replays must equal the eager query bit for bit, also after the host inputs
change between replays."""
import numpy as np
import pytest
import torch

import cs_workloads as W
from _helpers import bits16, cuda
from paper_2607_19547_gb300.pipeline import ComposedQuery, GraphedQuery, QueryShape, compose_from_host

pytestmark = pytest.mark.gpu


def _setup(w, seed):
    x = W.make_inputs(w, seed=seed, device="cuda")
    loc, glo = W.coordinates(w)
    pl, pg = cuda(loc), cuda(glo)
    cand = slice(w.cand0, w.cand0 + w.n_cand)
    import paper_2607_19547_gb300 as cs
    fresh = torch.empty_like(x["k_fresh_local"])
    cs.cs_rebase_keys(x["k_fresh_local"][None], pl[cand].contiguous(), pg[cand].contiguous(),
                      k_out=fresh[None])
    host = {"k": x["k"].cpu().pin_memory(), "v": x["v"].cpu().pin_memory(),
            "q": x["q"].cpu().pin_memory(), "k_fresh": fresh.cpu().pin_memory()}
    dev = {"k": torch.empty_like(x["k"]), "v": torch.empty_like(x["v"]), "q": torch.empty_like(x["q"]),
           "k_fresh": torch.empty_like(fresh), "pos_local": pl, "pos_global": pg}
    shape = QueryShape(n_layers=w.n_layers, T=w.T, hq=w.hq, hkv=w.hkv, cand0=w.cand0,
                       n_cand=w.n_cand, k=w.k, suffix=w.suffix, score_layer=w.score_layer)
    return shape, host, dev


def _out_host(q, w):
    return {"o": torch.empty(q.out.shape, dtype=q.out.dtype).pin_memory(),
            "qpos": torch.empty(w.M, dtype=torch.int32).pin_memory()}


@pytest.mark.parametrize("name", ["tiny_f32", "qwen3b_4x1024"])
def test_graph_replay_equals_eager(cslib, name):
    w = W.CONFIGS[name]
    shape, host, dev = _setup(w, 21)
    # eager reference on its own buffers
    qe = ComposedQuery(shape, w.torch_dtype)
    eager = _out_host(qe, w)
    dev_e = {k: (v.clone() if k in ("k", "v", "q", "k_fresh") else v) for k, v in dev.items()}
    compose_from_host(qe, host, dev_e, eager)
    torch.cuda.synchronize()
    # graph
    qg = ComposedQuery(shape, w.torch_dtype)
    got = _out_host(qg, w)
    gq = GraphedQuery(qg, host, dev, got)
    for _ in range(2):
        for t in got.values():
            t.zero_()
        gq.replay()
        torch.cuda.synchronize()
        cslib.cs_sync_status()
        assert np.array_equal(got["qpos"].numpy(), eager["qpos"].numpy())
        if w.dtype == "bf16":
            assert np.array_equal(bits16(got["o"]), bits16(eager["o"]))
        else:
            assert torch.equal(got["o"], eager["o"])
    # new queries in the same host buffer: the replay reads them
    host["q"].copy_(torch.randn(host["q"].shape, generator=torch.Generator().manual_seed(3)).to(host["q"].dtype))
    gq.replay()
    compose_from_host(qe, host, dev_e, eager)
    torch.cuda.synchronize()
    if w.dtype == "bf16":
        assert np.array_equal(bits16(got["o"]), bits16(eager["o"]))
    else:
        assert torch.equal(got["o"], eager["o"])


@pytest.mark.parametrize("name,policy,group,bounds", [
    ("tiny_f32", "3axis", 6, None), ("qwen3b_4x1024", "3axis", 6, None),
    ("qwen3b_4x1024", "scalar1d", 5, None), ("qwen3b_4x1024", "naive", 36, None),
    ("qwen3b_4x1024", "3axis", 4, [0, 2, 3, 20, 35, 36])])
def test_pipelined_query_equals_eager(cslib, name, policy, group, bounds):
    """Uploads, kernels and downloads overlapped layer group by layer group (one graph) give the
    eager query's result bit for bit."""
    from paper_2607_19547_gb300.pipeline import PipelinedQuery
    w = W.CONFIGS[name]
    shape, host, dev = _setup(w, 31)
    qe = ComposedQuery(shape, w.torch_dtype)
    eager = _out_host(qe, w)
    dev_e = {k: (v.clone() if k in ("k", "v", "q", "k_fresh") else v) for k, v in dev.items()}
    compose_from_host(qe, host, dev_e, eager, policy=policy)
    torch.cuda.synchronize()
    qp = ComposedQuery(shape, w.torch_dtype)
    got = _out_host(qp, w)
    pq = PipelinedQuery(qp, host, dev, got, group_layers=group, policy=policy, bounds=bounds)
    for _ in range(2):
        for t in got.values():
            t.zero_()
        pq.replay()
        torch.cuda.synchronize()
        cslib.cs_sync_status()
        assert np.array_equal(got["qpos"].numpy(), eager["qpos"].numpy())
        if w.dtype == "bf16":
            assert np.array_equal(bits16(got["o"]), bits16(eager["o"]))
        else:
            assert torch.equal(got["o"], eager["o"])


@pytest.mark.parametrize("name,n_slots,policy", [("tiny_f32", 2, "3axis"),
                                                 ("qwen3b_4x1024", 2, "3axis"),
                                                 ("qwen3b_4x1024", 4, "3axis"),
                                                 ("qwen3b_4x1024", 2, "scalar1d"),
                                                 ("qwen3b_4x1024", 3, "naive")])
def test_query_stream_equals_eager(cslib, name, n_slots, policy):
    """A stream of queries with n_slots in flight: every slot's result equals the eager query on
    that slot's host inputs, bit for bit, while the other slots' queries overlap it."""
    from paper_2607_19547_gb300.pipeline import QueryStream
    w = W.CONFIGS[name]
    shape, host0, dev = _setup(w, 41)
    # the other slots serve other queries (new q rows) over the same cache
    hosts = [host0]
    for s in range(1, n_slots):
        h = dict(host0)
        h["q"] = torch.randn(host0["q"].shape, generator=torch.Generator().manual_seed(5 + s)).to(
            host0["q"].dtype).pin_memory()
        hosts.append(h)
    expect = []
    for h in hosts:
        qe = ComposedQuery(shape, w.torch_dtype)
        eo = _out_host(qe, w)
        dev_e = {k: (v.clone() if k in ("k", "v", "q", "k_fresh") else v) for k, v in dev.items()}
        compose_from_host(qe, h, dev_e, eo, policy=policy)
        torch.cuda.synchronize()
        expect.append(eo)
    qs = QueryStream(shape, w.torch_dtype, hosts, dev["pos_local"], dev["pos_global"],
                     n_slots=n_slots, policy=policy)
    for n in (n_slots, 2 * n_slots + 1):
        for s in range(n_slots):
            for t in qs.out_host(s).values():
                t.zero_()
        qs.run(n)
        torch.cuda.synchronize()
        cslib.cs_sync_status()
        for s in range(n_slots):
            got, eo = qs.out_host(s), expect[s]
            assert np.array_equal(got["qpos"].numpy(), eo["qpos"].numpy())
            if w.dtype == "bf16":
                assert np.array_equal(bits16(got["o"]), bits16(eo["o"]))
            else:
                assert torch.equal(got["o"], eo["o"])
