"""Re-base (Eq. 3) on the GPU against the oracle: bf16 outputs must equal the oracle's
correctly rounded result bit for bit (and sit within 2e-2 of the exact rotation);
fp32 outputs within 1e-5 of the exact rotation."""
import numpy as np
import pytest
import torch

import cs_workloads as W
import oracle as O
from _helpers import TOL, bits16, cuda, f64

pytestmark = pytest.mark.gpu


def _check(cs, k_dev, loc, glo, dtype_name, tokens=None, out_of_place=False, layer_pad=0,
           allowed_mismatch=0.0):
    """Runs cs_rebase_keys on k_dev and compares (optionally sampled tokens) with the oracle.

    allowed_mismatch: fraction of bf16 elements that may differ by one unit in the last
    place; only needed where the oracle's own fp64 angle fl64(Delta * theta_i) carries an
    error of |Delta * theta_i| * 2^-53 comparable to the distance to a rounding midpoint."""
    before = f64(k_dev)
    L, T, H, D = k_dev.shape
    if layer_pad:
        buf = torch.zeros((L, T + layer_pad, H, D), dtype=k_dev.dtype, device="cuda")
        buf[:, :T] = k_dev
        k_dev = buf[:, :T]
    pl, pg = cuda(loc), cuda(glo)
    if out_of_place:
        out = torch.full_like(k_dev, float("nan")) if not layer_pad else \
            torch.full((L, T + layer_pad, H, D), float("nan"), dtype=k_dev.dtype,
                       device="cuda")[:, :T]
        res = cs.cs_rebase_keys(k_dev, pl, pg, k_out=out)
        assert np.array_equal(f64(k_dev), before)          # input untouched
    else:
        res = cs.cs_rebase_keys(k_dev, pl, pg)
    cs.cs_sync_status()
    sel = slice(None) if tokens is None else tokens
    exp_r, exp_x = O.rebase(before[:, sel], loc[sel], glo[sel], dtype_name)
    got = res[:, sel] if tokens is None else res[:, torch.as_tensor(tokens, device="cuda")]
    got64 = f64(got)
    assert np.max(np.abs(got64 - exp_x)) <= TOL[dtype_name]
    if dtype_name == "bf16":
        gb, eb = bits16(got), O.bf16_bits(exp_r)
        diff = gb != eb
        mism = int(np.sum(diff))
        assert mism <= allowed_mismatch * gb.size, \
            f"{mism} bf16 elements differ from the correctly rounded rotation"
        if mism:
            steps = np.abs(gb[diff].astype(np.int32) - eb[diff].astype(np.int32))
            assert steps.max() == 1
    return res


def test_tiny_f32_config(cslib):
    w = W.CONFIGS["tiny_f32"]
    x = W.make_inputs(w, seed=0, device="cuda")
    loc, glo = W.coordinates(w)
    _check(cslib, x["k"], loc, glo, "f32")
    _check(cslib, W.make_inputs(w, seed=1, device="cuda")["k"], loc, glo, "f32", out_of_place=True)


def test_qwen3b_4x1024_full(cslib):
    w = W.CONFIGS["qwen3b_4x1024"]
    x = W.make_inputs(w, seed=0, device="cuda")
    loc, glo = W.coordinates(w)
    _check(cslib, x["k"], loc, glo, "bf16")


@pytest.mark.parametrize("H", [1, 2, 4, 7])
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_random_coordinates_ragged(cslib, H, dtype):
    T, L = 333, 3
    g = torch.Generator(device="cuda").manual_seed(100 + H)
    k = torch.randn((L, T, H, 128), generator=g, device="cuda").to(dtype)
    loc, glo = W.random_coordinates(T, seed=H, max_coord=100000)
    glo[::7] = loc[::7]                         # some tokens do not move
    glo[1::5, 1] = loc[1::5, 1]                 # some move on two axes only
    name = "bf16" if dtype == torch.bfloat16 else "f32"
    _check(cslib, k.clone(), loc, glo, name)
    _check(cslib, k.clone(), loc, glo, name, out_of_place=True)
    _check(cslib, k.clone(), loc, glo, name, layer_pad=5)


def test_extreme_deltas(cslib):
    T = 64
    k = torch.randn((2, T, 2, 128), device="cuda").to(torch.bfloat16)
    loc = np.zeros((T, 3), np.int32)
    glo = np.zeros((T, 3), np.int32)
    big = np.array([1, -1, 2 ** 20, -(2 ** 20), 2 ** 24, 123456789, -987654321, 2 ** 30 - 1])
    for a in range(3):
        glo[:, a] = np.resize(big, T) // (a + 1)
    # angles up to ~1e9 rad: the oracle's fp64 angle is only good to ~1e-7 rad here
    _check(cslib, k, loc, glo, "bf16", allowed_mismatch=1e-3)


def test_delta_zero_is_identity_bit_for_bit(cslib):
    w = W.CONFIGS["qwen3b_4x1024"].with_(n_layers=3)
    x = W.make_inputs(w, seed=5, device="cuda")
    loc, _ = W.coordinates(w)
    before = bits16(x["k"])
    cslib.cs_rebase_keys(x["k"], cuda(loc), cuda(loc))
    cslib.cs_sync_status()
    assert np.array_equal(bits16(x["k"]), before)
    out = torch.zeros_like(x["k"])
    cslib.cs_rebase_keys(x["k"], cuda(loc), cuda(loc), k_out=out)
    cslib.cs_sync_status()
    assert np.array_equal(bits16(out), before)


def test_unmoved_tokens_untouched_in_place(cslib):
    w = W.CONFIGS["qwen3b_4x1024"].with_(n_layers=2)
    x = W.make_inputs(w, seed=6, device="cuda")
    loc, glo = W.coordinates(w)
    before = bits16(x["k"])
    cslib.cs_rebase_keys(x["k"], cuda(loc), cuda(glo))
    cslib.cs_sync_status()
    after = bits16(x["k"])
    assert np.array_equal(after[:, :w.cand0], before[:, :w.cand0])
    assert np.mean(after[:, w.cand0:] != before[:, w.cand0:]) > 0.5


@pytest.mark.parametrize("name", ["qwen3b_16x1024_q64", "qwen3b_64x1024_r15", "qwen7b_32x2048"])
def test_large_configs_sampled_tokens(cslib, name):
    w = W.CONFIGS[name]
    x = W.make_inputs(w, seed=0, device="cuda")
    loc, glo = W.coordinates(w)
    tokens = W.sample_rows(w.T, 600, seed=3)
    before = f64(x["k"][:, torch.as_tensor(tokens, device="cuda")])
    cslib.cs_rebase_keys(x["k"], cuda(loc), cuda(glo))
    cslib.cs_sync_status()
    got = x["k"][:, torch.as_tensor(tokens, device="cuda")]
    exp_r, exp_x = O.rebase(before, loc[tokens], glo[tokens], "bf16")
    assert np.max(np.abs(f64(got) - exp_x)) <= TOL["bf16"]
    assert int(np.sum(bits16(got) != O.bf16_bits(exp_r))) == 0
