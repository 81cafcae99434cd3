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


@pytest.mark.parametrize("H", [8, 16, 32])
def test_many_kv_heads_bf16(cslib, H):
    """Up to the 32 kv heads the bf16 kernel accepts: one token per block, 1-4 layer slots."""
    T, L = 37, 5
    g = torch.Generator(device="cuda").manual_seed(500 + H)
    k = torch.randn((L, T, H, 128), generator=g, device="cuda").to(torch.bfloat16)
    loc, glo = W.random_coordinates(T, seed=H, max_coord=4000)
    glo[::5] = loc[::5]
    _check(cslib, k.clone(), loc, glo, "bf16")
    _check(cslib, k.clone(), loc, glo, "bf16", out_of_place=True)


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


def _hard_pairs(L, T, H, loc, glo, seed):
    """bf16 keys [L, T, H, 128] whose rotations often land where the fp32 fast path cannot
    decide the bf16 rounding: exact zeros, subnormal and tiny values, values near the top of
    the bf16 range, and pairs chosen so that one output of the rotation nearly cancels."""
    rng = np.random.default_rng(seed)
    shape = (L, T, H, 64)
    x = rng.standard_normal(shape)
    y = rng.standard_normal(shape)
    cls = rng.integers(0, 8, size=shape)

    def mag(lo, hi):
        return np.exp2(rng.uniform(lo, hi, size=shape)) * rng.choice([-1.0, 1.0], size=shape)

    theta = O.rope_theta(1e6, 128)
    ang = (glo - loc).astype(np.float64)[:, O.axis_of_pair((16, 24, 24))] * theta   # [T, 64]
    c, s = np.cos(ang)[None, :, None, :], np.sin(ang)[None, :, None, :]
    with np.errstate(divide="ignore", invalid="ignore"):
        cancel1 = np.clip(np.where(np.abs(s) > 1e-6, x * c / s, 0.0), -1e30, 1e30)    # x c - y s ~ 0
        cancel2 = np.clip(np.where(np.abs(s) > 1e-6, -y * c / s, 0.0), -1e30, 1e30)   # y c + x s ~ 0
    x = np.where(cls == 0, 0.0, x)
    y = np.where(cls == 0, 0.0, y)
    y = np.where(cls == 1, 0.0, y)
    x = np.where(cls == 2, mag(-133, -126), x)
    y = np.where(cls == 2, mag(-133, -118), y)
    x = np.where(cls == 3, mag(100, 127.9), x)
    y = np.where(cls == 3, mag(100, 127.9), y)
    y = np.where(cls == 4, cancel1, y)
    x = np.where(cls == 5, cancel2, x)
    k = np.concatenate([x, y], axis=-1)
    return torch.tensor(k, dtype=torch.float64).to(torch.float32).to(torch.bfloat16)


@pytest.mark.parametrize("H", [1, 2, 4])
@pytest.mark.parametrize("out_of_place", [False, True])
def test_rounding_hard_cases_bit_exact(cslib, H, out_of_place):
    """Most slices here fail the fp32 rounding test, so the per-warp redo queue fills and is
    drained inside the layer loop many times; every output must still be the correctly
    rounded rotation, bit for bit (the max-abs bound does not apply to keys near 2^127)."""
    L, T = 16, 101
    loc, glo = W.random_coordinates(T, seed=40 + H, max_coord=3000)
    glo[::9] = loc[::9]
    k = _hard_pairs(L, T, H, loc, glo, seed=H).cuda()
    before = f64(k)
    assert np.all(np.isfinite(before))
    if out_of_place:
        res = cslib.cs_rebase_keys(k, cuda(loc), cuda(glo), k_out=torch.empty_like(k))
    else:
        res = cslib.cs_rebase_keys(k, cuda(loc), cuda(glo))
    cslib.cs_sync_status()
    exp_r, _ = O.rebase(before, loc, glo, "bf16")
    # an exactly zero rotation may come out as +0 or -0: compare zeros by value
    gb = np.where(bits16(res) == 0x8000, 0, bits16(res))
    eb = np.where(O.bf16_bits(exp_r) == 0x8000, 0, O.bf16_bits(exp_r))
    bad = gb != eb
    assert int(np.sum(bad)) == 0, (int(np.sum(bad)), gb[bad][:8], eb[bad][:8],
                                   before[..., :64][bad[..., :64]][:8],
                                   before[..., 64:][bad[..., :64]][:8])


def test_rounding_hard_cases_f32(cslib):
    """fp32 storage on the same hard inputs: within 2^-22 relative (plus an absolute 2^-140
    for subnormal results) of the exact rotation, and the infinity where it overflows."""
    L, T, H = 6, 77, 2
    loc, glo = W.random_coordinates(T, seed=77, max_coord=3000)
    k = _hard_pairs(L, T, H, loc, glo, seed=9).to(torch.float32).cuda()
    before = f64(k)
    res = cslib.cs_rebase_keys(k, cuda(loc), cuda(glo))
    cslib.cs_sync_status()
    exact = O.rebase_f64(before, loc, glo)
    expect = np.where(np.abs(exact) >= 2.0 ** 128 - 2.0 ** 103, np.copysign(np.inf, exact), exact)
    got = f64(res)
    inf = np.isinf(expect)
    assert np.array_equal(got[inf], expect[inf])
    err = np.abs(got[~inf] - expect[~inf])
    assert np.all(err <= np.abs(expect[~inf]) * 2.0 ** -22 + 2.0 ** -140)
