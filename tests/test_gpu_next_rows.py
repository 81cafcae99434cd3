"""The rows built after the four-step path: scatter-back of the repaired rows, the
scalar-1D and naive re-base policies, and the attention part of the shallow recompute,
each on the GPU against the oracle on the same seeded inputs."""
import numpy as np
import pytest
import torch

import cs_workloads as W
import oracle as O
from _helpers import TOL, bits16, cuda, f64
from paper_2607_19547_gb300.pipeline import ComposedQuery, QueryShape

pytestmark = pytest.mark.gpu


def _shape(w):
    return QueryShape(n_layers=w.n_layers, T=w.T, hq=w.hq, hkv=w.hkv, cand0=w.cand0,
                      n_cand=w.n_cand, k=w.k, suffix=w.suffix, score_layer=w.score_layer)


@pytest.mark.parametrize("dtype,H,n", [(torch.bfloat16, 2, 37), (torch.bfloat16, 4, 1),
                                       (torch.float32, 1, 64)])
def test_scatter_rows_bit_exact(cslib, dtype, H, n):
    g = torch.Generator().manual_seed(n)
    L, T = 3, 300
    cache = torch.randn(L, T, H, 128, generator=g).to(dtype)
    rows = torch.randn(L, n, H, 128, generator=g).to(dtype)
    idx = np.sort(np.random.default_rng(n).choice(T, n, replace=False)).astype(np.int32)
    exp = O.scatter_rows(f64(cache), f64(rows), idx)
    dc = cache.cuda()
    cslib.cs_scatter_rows(dc, rows.cuda(), cuda(idx))
    cslib.cs_sync_status()
    assert np.array_equal(f64(dc), exp)


def test_scatter_rows_strided_cache_and_bad_index(cslib):
    """A cache with a longer layer stride (a preallocated buffer) and one index out of range:
    the other rows land, the bad one is skipped and reported."""
    g = torch.Generator().manual_seed(5)
    L, T, H = 2, 50, 2
    buf = torch.randn(L, T + 14, H, 128, generator=g).to(torch.bfloat16)
    full = buf.cuda()
    cache = full[:, :T]
    before = bits16(buf)
    rows = torch.randn(L, 3, H, 128, generator=g).to(torch.bfloat16)
    idx = np.array([4, 9, T + 3], np.int32)
    cslib.cs_scatter_rows(cache, rows.cuda(), cuda(idx))
    with pytest.raises(cslib.CsError) as e:
        cslib.cs_sync_status()
    assert e.value.status == cslib.CS_ERR_DEVICE_ARG
    got = bits16(cache.contiguous())
    assert np.array_equal(got[:, 4], bits16(rows[:, 0])) and np.array_equal(got[:, 9], bits16(rows[:, 1]))
    untouched = np.setdiff1d(np.arange(T), [4, 9])
    assert np.array_equal(got[:, untouched], before[:, :T][:, untouched])
    assert np.array_equal(bits16(full)[:, T:], before[:, T:])   # nothing written past T
    cslib.cs_sync_status()                                      # the status word was cleared


@pytest.mark.parametrize("name", ["tiny_f32", "qwen3b_4x1024"])
def test_scalar1d_policy_matches_oracle(cslib, name):
    w = W.CONFIGS[name]
    x = W.make_inputs(w, seed=1, device="cuda")
    loc, _ = W.coordinates(w)
    layers = [0, w.n_layers - 1] if w.n_layers > 1 else [0]
    stored = {l: f64(x["k"][l]) for l in layers}
    q = ComposedQuery(_shape(w), w.torch_dtype)
    fresh = x["k_fresh_local"]
    out, qpos = q.step(x["k"], x["v"], x["q"], fresh, cuda(loc), None, policy="scalar1d")
    cslib.cs_sync_status()
    tgt = O.scalar1d_targets(w.T)
    for l in layers:
        exp, _ = O.rebase(stored[l][None], loc, tgt, w.dtype)
        if w.dtype == "bf16":
            assert np.array_equal(bits16(x["k"][l]), O.bf16_bits(exp[0]))
        else:
            assert np.max(np.abs(f64(x["k"][l]) - exp[0])) <= TOL["f32"]
    # the selection is taken on the scalar-re-based score-layer keys, stage-wise
    cand = slice(w.cand0, w.cand0 + w.n_cand)
    score = O.score_f32_canonical(f64(fresh).astype(np.float32),
                                  f64(x["k"][w.score_layer, cand]).astype(np.float32))
    assert np.array_equal(q.score.cpu().numpy().view(np.uint32), score.view(np.uint32))
    sel = O.select_topk(score, w.k, w.cand0)
    assert np.array_equal(qpos.cpu().numpy()[:w.k], sel)


def test_naive_policy_keeps_stored_keys(cslib):
    w = W.CONFIGS["qwen3b_4x1024"]
    x = W.make_inputs(w, seed=2, device="cuda")
    loc, glo = W.coordinates(w)
    before = bits16(x["k"])
    q = ComposedQuery(_shape(w), w.torch_dtype)
    q.step(x["k"], x["v"], x["q"], x["k_fresh_local"], cuda(loc), cuda(glo), policy="naive")
    cslib.cs_sync_status()
    assert np.array_equal(bits16(x["k"]), before)


@pytest.mark.parametrize("name", ["tiny_f32", "qwen3b_4x1024"])
def test_naive_policy_end_to_end_matches_oracle(cslib, name):
    """Table 1's naive concatenation: the stored keys stay at their chunk-local positions.
    Score, selection and the attention of sampled rows equal the oracle's on the un-rebased
    cache, with the fresh keys at global coordinates as the recompute would give them."""
    w = W.CONFIGS[name]
    x = W.make_inputs(w, seed=8, device="cuda")
    loc, glo = W.coordinates(w)
    cand = slice(w.cand0, w.cand0 + w.n_cand)
    layers = [0, w.n_layers - 1] if w.n_layers > 1 else [0]
    stored_k = {l: f64(x["k"][l]) for l in layers}
    k_score = f64(x["k"][w.score_layer, cand])
    fresh_local = f64(x["k_fresh_local"])
    fresh = torch.empty_like(x["k_fresh_local"])
    cslib.cs_rebase_keys(x["k_fresh_local"][None], cuda(loc[cand]), cuda(glo[cand]),
                         k_out=fresh[None])
    q = ComposedQuery(_shape(w), w.torch_dtype)
    out, qpos = q.step(x["k"], x["v"], x["q"], fresh, cuda(loc), cuda(glo), policy="naive")
    cslib.cs_sync_status()
    # the oracle: its own fresh keys at global coordinates, the stored keys as they are
    kf, _ = O.rebase(fresh_local[None], loc[cand], glo[cand], w.dtype)
    score = O.score_f32_canonical(kf[0].astype(np.float32), k_score.astype(np.float32))
    assert np.array_equal(q.score.cpu().numpy().view(np.uint32), score.view(np.uint32))
    sel = O.select_topk(score, w.k, w.cand0)
    exp_qpos = np.concatenate([sel, np.arange(w.T - w.suffix, w.T)]).astype(np.int32)
    assert np.array_equal(qpos.cpu().numpy(), exp_qpos)
    rows = W.sample_rows(w.M, 32, seed=10)
    for l in layers:
        eo, _ = O.repair_attention(f64(x["q"][l])[None][:, rows], stored_k[l][None],
                                   f64(x["v"][l])[None], exp_qpos[rows])
        go = f64(out[l][torch.as_tensor(rows, device="cuda")])[None]
        assert np.max(np.abs(go - eo)) <= TOL[w.dtype]


def test_pipeline_with_scatter_back_matches_oracle(cslib):
    """Fresh K/V of the repaired rows go into the cache before the attention: the attention of
    sampled rows equals the oracle's over the oracle-composed cache with those rows replaced."""
    w = W.CONFIGS["qwen3b_4x1024"]
    x = W.make_inputs(w, seed=3, device="cuda")
    loc, glo = W.coordinates(w)
    g = torch.Generator().manual_seed(11)
    k_rows = torch.randn(w.n_layers, w.k, w.hkv, 128, generator=g).to(torch.bfloat16)
    v_rows = torch.randn(w.n_layers, w.k, w.hkv, 128, generator=g).to(torch.bfloat16)
    layers = [0, w.n_layers - 1]
    stored_k = {l: f64(x["k"][l]) for l in layers}
    stored_v = {l: f64(x["v"][l]) for l in layers}
    q = ComposedQuery(_shape(w), w.torch_dtype)
    out, qpos = q.step(x["k"], x["v"], x["q"], x["k_fresh_local"], cuda(loc), cuda(glo),
                       fresh_kv=(k_rows.cuda(), v_rows.cuda()))
    cslib.cs_sync_status()
    sel = qpos.cpu().numpy()[:w.k]
    rows = W.sample_rows(w.M, 32, seed=4)
    for l in layers:
        k_l, _ = O.rebase(stored_k[l][None], loc, glo, "bf16")
        k_l = O.scatter_rows(k_l, f64(k_rows[l])[None], sel)
        v_l = O.scatter_rows(stored_v[l][None], f64(v_rows[l])[None], sel)
        # the cache now holds exactly the scattered rows
        assert np.array_equal(bits16(x["k"][l][torch.as_tensor(sel, device="cuda").long()]),
                              bits16(k_rows[l]))
        eo, _ = O.repair_attention(f64(x["q"][l])[None][:, rows], k_l, v_l, qpos.cpu().numpy()[rows])
        go = f64(out[l][torch.as_tensor(rows, device="cuda")])[None]
        assert np.max(np.abs(go - eo)) <= TOL["bf16"]


@pytest.mark.parametrize("name", ["tiny_f32", "qwen3b_4x1024"])
def test_shallow_recompute_attention_matches_oracle(cslib, name):
    """Every candidate as a query row over the first two layers (Eq. 6's 2 c_a |C| T term)."""
    w = W.CONFIGS[name]
    x = W.make_inputs(w, seed=6, device="cuda")
    nl = min(2, w.n_layers)
    g = torch.Generator().manual_seed(12)
    q_cand = torch.randn(nl, w.n_cand, w.hq, 128, generator=g).to(w.torch_dtype).cuda()
    q = ComposedQuery(_shape(w), w.torch_dtype)
    o = q.shallow_recompute(q_cand, x["k"], x["v"])
    cslib.cs_sync_status()
    assert o.shape == (nl, w.n_cand, w.hq, 128)
    pos = np.arange(w.cand0, w.cand0 + w.n_cand, dtype=np.int32)
    rows = W.sample_rows(w.n_cand, min(48, w.n_cand), seed=7)
    for l in range(nl):
        eo, _ = O.repair_attention(f64(q_cand[l])[None][:, rows], f64(x["k"][l])[None],
                                   f64(x["v"][l])[None], pos[rows])
        go = f64(o[l][torch.as_tensor(rows, device="cuda")])[None]
        assert np.max(np.abs(go - eo)) <= TOL[w.dtype]
