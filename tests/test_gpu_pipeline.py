"""The whole composition query (re-base -> score -> select -> repair attention) on the
GPU against the oracle run independently on the same seeded inputs.

Each side re-bases the stored keys and the fresh keys with its own code; the
re-based bf16 keys are the correctly rounded rotation on both sides, the score is
defined in one fp32 order, so the selected indices must agree bit for bit."""
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


@pytest.mark.parametrize("name", list(W.CONFIGS))
def test_pipeline_matches_oracle(cslib, name):
    w = W.CONFIGS[name]
    x = W.make_inputs(w, seed=0, device="cuda")
    loc, glo = W.coordinates(w)
    dname = w.dtype
    cand = slice(w.cand0, w.cand0 + w.n_cand)
    # ---- oracle inputs: exact copies of the stored tensors, taken before the GPU runs
    k_score_layer = f64(x["k"][w.score_layer, cand])
    fresh_local = f64(x["k_fresh_local"])
    # sampled layers: the first, the score layer, the quarters and the last
    L = w.n_layers
    layers = sorted({0, w.score_layer, L // 4, L // 2, (3 * L) // 4, L - 1})
    k_stored = {l: f64(x["k"][l]) for l in layers}
    # ---- GPU: fresh keys at global coordinates (the shallow recompute's output) ...
    fresh = torch.empty_like(x["k_fresh_local"])
    cslib.cs_rebase_keys(x["k_fresh_local"][None], cuda(loc[cand]), cuda(glo[cand]),
                         k_out=fresh[None])
    # ... then the four calls
    q = ComposedQuery(_shape(w), w.torch_dtype)
    out, qpos = q.step(x["k"], x["v"], x["q"], fresh, cuda(loc), cuda(glo))
    cslib.cs_sync_status()
    # ---- oracle, independently
    kc_r, _ = O.rebase(k_score_layer[None], loc[cand], glo[cand], dname)
    kf_r, _ = O.rebase(fresh_local[None], loc[cand], glo[cand], dname)
    score = O.score_f32_canonical(kf_r[0].astype(np.float32), kc_r[0].astype(np.float32))
    sel = O.select_topk(score, w.k, w.cand0)
    exp_qpos = np.concatenate([sel, np.arange(w.T - w.suffix, w.T)]).astype(np.int32)
    # the stages
    if dname == "bf16":
        assert np.array_equal(bits16(x["k"][w.score_layer, cand]), O.bf16_bits(kc_r[0]))
        assert np.array_equal(bits16(fresh), O.bf16_bits(kf_r[0]))
    got_score = q.score.cpu().numpy()
    assert np.array_equal(got_score.view(np.uint32), score.view(np.uint32))
    got_qpos = qpos.cpu().numpy()
    assert np.array_equal(got_qpos, exp_qpos), \
        f"{np.sum(got_qpos != exp_qpos)} selected indices differ"
    # attention over the composed cache, oracle fed its own re-based keys of the sampled layers
    rows = W.sample_rows(w.M, 256 if w.T > 5000 else w.M, seed=9)
    for l in layers:
        k_l, _ = O.rebase(k_stored[l][None], loc, glo, dname)
        v_l = f64(x["v"][l])[None]
        q_l = f64(x["q"][l])[None][:, rows]
        eo, _ = O.repair_attention(q_l, k_l, v_l, exp_qpos[rows])
        go = f64(out[l][torch.as_tensor(rows, device="cuda")])[None]
        err = np.max(np.abs(go - eo))
        assert err <= TOL[dname], f"layer {l}: max abs error {err}"


def test_bench_workload_every_layer(cslib):
    """The bench workload (64 chunks x 1024 tokens, rho 0.15) end to end, its attention checked
    on every one of the 36 layers against the oracle run on that layer's own re-based keys, on 32
    seeded rows (first and last included) per layer."""
    w = W.CONFIGS["qwen3b_64x1024_r15"]
    x = W.make_inputs(w, seed=3, device="cuda")
    loc, glo = W.coordinates(w)
    cand = slice(w.cand0, w.cand0 + w.n_cand)
    k_stored = x["k"].clone()                     # the stored keys, before the in-place re-base
    fresh = torch.empty_like(x["k_fresh_local"])
    cslib.cs_rebase_keys(x["k_fresh_local"][None], cuda(loc[cand]), cuda(glo[cand]),
                         k_out=fresh[None])
    q = ComposedQuery(_shape(w), w.torch_dtype)
    out, qpos = q.step(x["k"], x["v"], x["q"], fresh, cuda(loc), cuda(glo))
    cslib.cs_sync_status()
    # the selection, from the oracle's own re-base and score
    kc_r, _ = O.rebase(f64(k_stored[w.score_layer, cand])[None], loc[cand], glo[cand], w.dtype)
    kf_r, _ = O.rebase(f64(x["k_fresh_local"])[None], loc[cand], glo[cand], w.dtype)
    score = O.score_f32_canonical(kf_r[0].astype(np.float32), kc_r[0].astype(np.float32))
    exp_qpos = O.select_topk(score, w.k, w.cand0).astype(np.int32)
    assert np.array_equal(qpos.cpu().numpy(), exp_qpos)
    rows = W.sample_rows(w.M, 32, seed=13)
    rows_dev = torch.as_tensor(rows, device="cuda")
    worst = 0.0
    for l in range(w.n_layers):
        k_l, _ = O.rebase(f64(k_stored[l])[None], loc, glo, w.dtype)
        eo, _ = O.repair_attention(f64(x["q"][l])[None][:, rows], k_l, f64(x["v"][l])[None],
                                   exp_qpos[rows])
        err = float(np.max(np.abs(f64(out[l][rows_dev])[None] - eo)))
        worst = max(worst, err)
        assert err <= TOL[w.dtype], f"layer {l}: max abs error {err}"
    assert worst > 0.0          # the comparison ran on real values


@pytest.mark.parametrize("rho_bp", [0, 10000])
@pytest.mark.parametrize("base", ["tiny_f32", "qwen3b_4x1024"])
def test_pipeline_degenerate_rho(cslib, base, rho_bp):
    """The method's two ends, end to end: rho = 0 repairs no token (only the text-suffix rows
    query the cache), rho = 1 repairs every candidate.  Selection and attention against the
    oracle on the same inputs."""
    w = W.CONFIGS[base].with_(rho_bp=rho_bp, suffix=8, n_layers=min(3, W.CONFIGS[base].n_layers))
    assert w.k == (0 if rho_bp == 0 else w.n_cand)
    x = W.make_inputs(w, seed=17, device="cuda")
    loc, glo = W.coordinates(w)
    cand = slice(w.cand0, w.cand0 + w.n_cand)
    k_stored = f64(x["k"])
    fresh = torch.empty_like(x["k_fresh_local"])
    cslib.cs_rebase_keys(x["k_fresh_local"][None], cuda(loc[cand]), cuda(glo[cand]),
                         k_out=fresh[None])
    q = ComposedQuery(_shape(w), w.torch_dtype)
    out, qpos = q.step(x["k"], x["v"], x["q"], fresh, cuda(loc), cuda(glo))
    cslib.cs_sync_status()
    kc_r, _ = O.rebase(k_stored[w.score_layer, cand][None], loc[cand], glo[cand], w.dtype)
    kf_r, _ = O.rebase(f64(x["k_fresh_local"])[None], loc[cand], glo[cand], w.dtype)
    score = O.score_f32_canonical(kf_r[0].astype(np.float32), kc_r[0].astype(np.float32))
    sel = O.select_topk(score, w.k, w.cand0)
    exp_qpos = np.concatenate([sel, np.arange(w.T - w.suffix, w.T)]).astype(np.int32)
    if rho_bp == 10000:
        assert np.array_equal(sel, np.arange(w.cand0, w.cand0 + w.n_cand))
    assert np.array_equal(qpos.cpu().numpy(), exp_qpos)
    rows = W.sample_rows(w.M, 64, seed=19)
    k_r, _ = O.rebase(k_stored, loc, glo, w.dtype)
    eo, _ = O.repair_attention(f64(x["q"])[:, rows], k_r, f64(x["v"]), exp_qpos[rows])
    go = f64(out[:, torch.as_tensor(rows, device="cuda")])
    assert np.max(np.abs(go - eo)) <= TOL[w.dtype]
