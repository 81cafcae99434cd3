"""Host-side checks of the synthetic workloads: sizes, layout and determinism."""
import numpy as np
import pytest
import torch

import cs_workloads as W


@pytest.mark.parametrize("name,T,n_cand,k", [
    ("tiny_f32", 64, 32, 8),
    ("qwen3b_4x1024", 4104, 3072, 461),
    ("qwen3b_16x1024_q64", 16456, 15360, 2304),
    ("qwen3b_64x1024_r05", 65544, 64512, 3226),
    ("qwen3b_64x1024_r15", 65544, 64512, 9677),
    ("qwen3b_64x1024_r30", 65544, 64512, 19354),
    ("qwen7b_32x2048", 65544, 63488, 9524),
])
def test_config_sizes(name, T, n_cand, k):
    w = W.CONFIGS[name]
    assert (w.T, w.n_cand, w.k) == (T, n_cand, k)
    assert w.hq % w.hkv == 0


@pytest.mark.parametrize("name", list(W.CONFIGS))
def test_coordinate_layout(name):
    w = W.CONFIGS[name]
    loc, glo = W.coordinates(w)
    moved = np.any(loc != glo, axis=1)
    # prefix, chunk 0 and suffix stay; every later-chunk token moves
    assert not moved[:w.cand0].any()
    assert moved[w.cand0:w.prefix + w.t_vis].all()
    assert not moved[w.prefix + w.t_vis:].any()
    # chunks occupy non-overlapping global intervals on the temporal axis
    C = w.chunk_tokens
    for c in range(w.n_chunks - 1):
        a = glo[w.prefix + c * C: w.prefix + (c + 1) * C, 0]
        b = glo[w.prefix + (c + 1) * C: w.prefix + (c + 2) * C, 0]
        assert a.max() < b.min()
    # text tokens carry one scalar on all three axes
    for sl in (slice(0, w.prefix), slice(w.T - w.suffix, w.T)):
        assert (glo[sl, 0] == glo[sl, 1]).all() and (glo[sl, 1] == glo[sl, 2]).all()


def test_tiny_layout_is_single_video_shift():
    w = W.CONFIGS["tiny_f32"]
    loc, glo = W.coordinates(w)
    d = glo - loc
    assert (d[32:] == [2, 0, 0]).all() and (d[:32] == 0).all()
    assert loc[:, 0].max() == 1 and loc[:, 1:].max() == 3


def test_inputs_are_seeded_and_shaped():
    w = W.CONFIGS["tiny_f32"]
    a = W.make_inputs(w, seed=3)
    b = W.make_inputs(w, seed=3)
    c = W.make_inputs(w, seed=4)
    for key in a:
        assert torch.equal(a[key], b[key])
    assert not torch.equal(a["k"], c["k"])
    assert a["k"].shape == (1, 64, 1, 128) and a["q"].shape == (1, 8, 2, 128)
    assert a["k_fresh_local"].shape == (32, 1, 128)
    w3 = W.CONFIGS["qwen3b_4x1024"].with_(n_layers=2)
    x = W.make_inputs(w3, seed=0)
    assert x["k"].dtype == torch.bfloat16 and x["q"].shape == (2, 461, 16, 128)


def test_sample_rows_keeps_ends():
    r = W.sample_rows(1000, 50, seed=1)
    assert r[0] == 0 and r[-1] == 999 and len(r) == 50 and np.all(np.diff(r) > 0)
    assert list(W.sample_rows(5, 50, seed=1)) == [0, 1, 2, 3, 4]


def test_layer_subset_matches_full_draw():
    """Every layer has its own seed: a subset of layers is the same tensors as the full draw,
    and the fresh keys do not depend on which layers were asked for."""
    w = W.CONFIGS["qwen3b_4x1024"].with_(n_layers=3, n_chunks=2, grid_t=1, grid_h=4, grid_w=4)
    full = W.make_inputs(w, seed=5)
    sub = W.make_inputs(w, seed=5, layers=[2, 0])
    for key in ("k", "v", "q"):
        assert torch.equal(sub[key][0], full[key][2]) and torch.equal(sub[key][1], full[key][0])
    assert torch.equal(sub["k_fresh_local"], full["k_fresh_local"])
    assert not torch.equal(full["k"][0], full["k"][1])
