"""Pins of the CPU oracle against things other than itself.

Each test fixes the oracle to a closed form, an independent library routine
(math.cos/sin, numpy complex exponentials, torch's bf16 conversion, torch
SDPA), brute force on tiny inputs, or a figure printed in the paper
(tests/golden/paper_figures.json).  Each is chosen so that a plausible slip
(wrong theta schedule, wrong axis order, interleaved pairs, flipped rotation,
sign of Delta, dropped term, transposed operand, wrong tie-break) fails it.
"""
import math

import numpy as np
import pytest
import torch

import cs_workloads as W
import oracle as O

BASE = 1e6
SEC = (16, 24, 24)
D = 128


def unit(j):
    e = np.zeros(D)
    e[j] = 1.0
    return e


# ---------------------------------------------------------------- Eq. 2 ----

def test_theta_schedule_closed_form():
    th = O.rope_theta(BASE, D)
    assert th.shape == (64,)
    assert th[0] == 1.0
    # theta_i = 1e6^(-2i/128) = 10^(-3i/32)
    for i in (1, 16, 40, 63):
        assert th[i] == pytest.approx(10.0 ** (-3.0 * i / 32.0), rel=1e-14)
    assert th[16] == pytest.approx(10.0 ** -1.5, rel=1e-14)


def test_axis_assignment_matches_paper_sections(golden):
    sec = golden["model"]["mrope_sections"]
    sig = O.axis_of_pair(sec)
    assert list(np.bincount(sig)) == sec
    assert sig[0] == 0 and sig[15] == 0 and sig[16] == 1 and sig[39] == 1
    assert sig[40] == 2 and sig[63] == 2


@pytest.mark.parametrize("pair,axis", [(0, 0), (15, 0), (16, 1), (39, 1), (40, 2), (63, 2)])
def test_rotation_of_unit_vectors(pair, axis):
    p = np.array([3, 5, 7])
    ang = p[axis] * (10.0 ** (-3.0 * pair / 32.0))
    out = O.mrope_rotate(unit(pair), p, BASE, SEC)
    expect = np.zeros(D)
    expect[pair] = math.cos(ang)
    expect[pair + 64] = math.sin(ang)
    np.testing.assert_allclose(out, expect, atol=1e-15)
    out2 = O.mrope_rotate(unit(pair + 64), p, BASE, SEC)
    expect2 = np.zeros(D)
    expect2[pair] = -math.sin(ang)
    expect2[pair + 64] = math.cos(ang)
    np.testing.assert_allclose(out2, expect2, atol=1e-15)


def test_text_token_is_one_dimensional_rope_complex_form():
    """A text token (s, s, s) gets plain RoPE: z_i * exp(i s theta_i), z_i = x_i + i x_{i+64}."""
    rng = np.random.default_rng(1)
    x = rng.standard_normal((5, D))
    s = np.array([0, 1, 17, 999, 4103])
    pos = np.stack([s, s, s], axis=1)
    z = x[:, :64] + 1j * x[:, 64:]
    theta = np.array([BASE ** (-2.0 * i / D) for i in range(64)])
    zr = z * np.exp(1j * s[:, None] * theta[None, :])
    expect = np.concatenate([zr.real, zr.imag], axis=1)
    np.testing.assert_allclose(O.mrope_rotate(x, pos, BASE, SEC), expect, atol=1e-12)


# ---------------------------------------------------------------- Eq. 3 ----

def test_eq3_rebase_equals_rotation_at_target():
    """R(Delta) f(x, p) = f(x, p') for arbitrary coordinates."""
    rng = np.random.default_rng(2)
    T, H = 64, 3
    x = rng.standard_normal((T, H, D))
    p = rng.integers(0, 5000, size=(T, 3))
    pp = rng.integers(0, 5000, size=(T, 3))
    stored = O.mrope_rotate(x, p[:, None, :], BASE, SEC)
    joint = O.mrope_rotate(x, pp[:, None, :], BASE, SEC)
    moved = O.rebase_f64(stored, p, pp, BASE, SEC)
    assert np.max(np.abs(moved - joint)) < 1e-11
    # the wrong sign of Delta lands elsewhere
    wrong = O.rebase_f64(stored, pp, p, BASE, SEC)
    assert np.max(np.abs(wrong - joint)) > 0.1


def test_eq3_layer0_fidelity_within_table1(golden):
    """Table 1: at layer 0 the three-axis re-base reproduces the joint keys (rel MSE 3.6e-8)."""
    w = W.CONFIGS["qwen3b_4x1024"]
    loc, glo = W.coordinates(w)
    rng = np.random.default_rng(3)
    x = rng.standard_normal((w.T, 2, D))
    stored = O.mrope_rotate(x, loc[:, None, :], BASE, SEC)
    joint = O.mrope_rotate(x, glo[:, None, :], BASE, SEC)
    moved32 = O.round_to_storage(O.rebase_f64(stored, loc, glo, BASE, SEC), "f32")
    relmse = np.sum((moved32 - joint) ** 2) / np.sum(joint ** 2)
    assert relmse < golden["table1_layer0"]["three_axis_relmse"]


def test_rebase_delta_zero_is_bit_exact():
    rng = np.random.default_rng(4)
    k = O.round_to_bf16(rng.standard_normal((2, 16, 2, D)))
    pos = rng.integers(0, 100, size=(16, 3))
    r, _ = O.rebase(k, pos, pos, "bf16")
    assert np.array_equal(O.bf16_bits(r), O.bf16_bits(k))
    k32 = rng.standard_normal((2, 16, 2, D)).astype(np.float32).astype(np.float64)
    r32, _ = O.rebase(k32, pos, pos, "f32")
    assert np.array_equal(r32, k32)


def test_rebase_group_properties():
    rng = np.random.default_rng(5)
    T = 32
    x = rng.standard_normal((T, 2, D))
    p0 = rng.integers(-300, 300, size=(T, 3))
    p1 = rng.integers(-300, 300, size=(T, 3))
    p2 = rng.integers(-300, 300, size=(T, 3))
    two_step = O.rebase_f64(O.rebase_f64(x, p0, p1), p1, p2)
    one_step = O.rebase_f64(x, p0, p2)
    assert np.max(np.abs(two_step - one_step)) < 1e-12
    back = O.rebase_f64(O.rebase_f64(x, p0, p1), p1, p0)
    assert np.max(np.abs(back - x)) < 1e-12
    y = O.rebase_f64(x, p0, p1)
    nx = x[..., :64] ** 2 + x[..., 64:] ** 2
    ny = y[..., :64] ** 2 + y[..., 64:] ** 2
    np.testing.assert_allclose(ny, nx, rtol=1e-12)


def test_common_shift_keeps_attention_logits():
    """Moving every query and key by the same Delta leaves q.k unchanged (relative positions)."""
    rng = np.random.default_rng(6)
    T = 16
    q = rng.standard_normal((T, 1, D))
    k = rng.standard_normal((T, 1, D))
    p = rng.integers(0, 500, size=(T, 3))
    shift = np.array([[40, 7, 13]])
    qs = O.rebase_f64(q, p, p + shift)
    ks = O.rebase_f64(k, p, p + shift)
    np.testing.assert_allclose(qs[:, 0] @ ks[:, 0].T, q[:, 0] @ k[:, 0].T, atol=1e-10)


def test_scalar1d_reindex_is_not_three_axis(golden):
    """Sec. 2 / Table 1: the scalar re-index differs from the three-axis re-base.

    On the synthetic layout the layer-0 error ordering of Table 1 holds:
    three-axis (exact) < naive concatenation < scalar 1-D.
    """
    w = W.CONFIGS["qwen3b_4x1024"]
    loc, glo = W.coordinates(w)
    sc = O.scalar1d_targets(w.T)
    vis = slice(w.prefix, w.prefix + w.t_vis)
    # only the very first visual token, (P, P, P), keeps its coordinate
    assert np.any(sc[vis] != glo[vis], axis=1).sum() == w.t_vis - 1
    rng = np.random.default_rng(7)
    x = rng.standard_normal((w.T, 2, D))
    stored = O.mrope_rotate(x, loc[:, None, :], BASE, SEC)
    joint = O.mrope_rotate(x, glo[:, None, :], BASE, SEC)
    scalar = O.rebase_f64(stored, loc, sc, BASE, SEC)
    three = O.rebase_f64(stored, loc, glo, BASE, SEC)
    # the scalar result is exactly 1-D RoPE at the sequence slot
    np.testing.assert_allclose(scalar, O.mrope_rotate(x, sc[:, None, :], BASE, SEC), atol=1e-11)

    def relmse(a):
        return np.sum((a[vis] - joint[vis]) ** 2) / np.sum(joint[vis] ** 2)

    t1 = golden["table1_layer0"]
    assert relmse(three) < t1["three_axis_relmse"]
    assert relmse(stored) > 1e3 * t1["three_axis_relmse"]
    assert relmse(scalar) > relmse(stored)


# ------------------------------------------------------- bf16 rounding ----

def test_round_to_bf16_matches_torch_on_fp32_values():
    rng = np.random.default_rng(8)
    x = rng.standard_normal(200000).astype(np.float32) * np.float32(2.0) ** rng.integers(
        -30, 30, 200000).astype(np.float32)
    ours = O.bf16_bits(O.round_to_bf16(x.astype(np.float64)))
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ours, ref)


def test_round_to_bf16_ties_and_subnormals():
    base = np.array([1.0, 1.0078125, -3.0, 2.0 ** -126, 2.0 ** -130], dtype=np.float64)
    ulp = np.array([2.0 ** -7, 2.0 ** -7, 2.0 ** -6, 2.0 ** -133, 2.0 ** -133])
    mid = base + np.sign(base) * ulp / 2
    r = O.round_to_bf16(mid)
    # ties go to the even neighbour: 1.0 (even) stays, 1.0078125 (odd) goes up
    assert r[0] == 1.0
    assert r[1] == 1.0078125 + 2.0 ** -7
    assert r[2] == -3.0
    assert r[3] == 2.0 ** -126
    assert r[4] == 2.0 ** -130
    x32 = mid.astype(np.float32)
    ref = torch.from_numpy(x32).to(torch.bfloat16).double().numpy()
    np.testing.assert_array_equal(r, ref)


def test_round_to_bf16_brute_force_on_fp64_values():
    """Values between fp32 numbers: the nearest of the two bf16 neighbours, by exact distance."""
    rng = np.random.default_rng(9)
    x = rng.standard_normal(20000) * 10.0 ** rng.uniform(-5, 5, 20000)
    r = O.round_to_bf16(x)
    for xi, ri in zip(x[:2000], r[:2000]):
        b = int(O.bf16_bits(ri))
        cands = [O.bf16_from_bits(np.uint16(c)) for c in (b - 1, b, b + 1) if 0 <= c < 0xFFFF]
        d = [abs(xi - float(c)) for c in cands]
        assert abs(xi - ri) == min(d)


# ---------------------------------------------------------------- Eq. 5 ----

def test_score_small_integers():
    a = np.zeros((3, 256), np.float32)
    b = np.zeros((3, 256), np.float32)
    a[0, 0], b[0, 200] = 3.0, 4.0                 # 9 + 16
    a[1, :] = 1.0                                 # 256 ones
    a[2, 17], b[2, 17] = 0.5, -0.25               # 0.75^2
    s = O.score_f32_canonical(a, b)
    assert s.tolist() == [25.0, 256.0, 0.5625]
    assert np.all(O.score_f32_canonical(a, a) == 0)


def test_score_canonical_grouping_by_hand():
    """The fixed order differs from a left-to-right sum; expected values worked out by hand."""
    u = np.float32(2.0 ** -12)                    # u*u = 2^-24: half an fp32 ulp of 1
    a = np.zeros((2, 256), np.float32)
    b = np.zeros((2, 256), np.float32)
    # within one block: ((1 + 2^-24) + (2^-24 + 2^-24)) = 1 + 2^-23; a sequential sum gives 1
    a[0, 0], a[0, 1], a[0, 2], a[0, 3] = 1.0, u, u, u
    # across blocks (B = 32): block 1 and block 17 meet at m = 16 before meeting block 0
    a[1, 0], a[1, 8], a[1, 17 * 8] = 1.0, u, u
    s = O.score_f32_canonical(a, b)
    assert s[0] == np.float32(1.0 + 2.0 ** -23)
    assert s[1] == np.float32(1.0 + 2.0 ** -23)
    seq = np.float32(0)
    for qv in (a[0] * a[0]):
        seq = np.float32(seq + qv)
    assert seq == np.float32(1.0)


@pytest.mark.parametrize("E", [128, 256, 512, 384])
def test_score_canonical_close_to_fp64(E):
    rng = np.random.default_rng(E)
    a = O.round_to_bf16(rng.standard_normal((500, E)) * 3).astype(np.float32)
    b = O.round_to_bf16(rng.standard_normal((500, E))).astype(np.float32)
    s32 = O.score_f32_canonical(a, b).astype(np.float64)
    s64 = O.score_f64(a, b)
    np.testing.assert_allclose(s32, s64, rtol=2e-6)


# ------------------------------------------------------------ selection ----

def _brute_select(vals, k, base):
    items = sorted(range(len(vals)), key=lambda i: (-vals[i], i))
    return sorted(base + i for i in items[:k])


@pytest.mark.parametrize("seed", range(6))
def test_select_matches_brute_force_with_ties(seed):
    rng = np.random.default_rng(seed)
    n = int(rng.integers(1, 400))
    vals = rng.choice(np.array([0.0, 0.5, 1.0, 2.0, 3.5, 100.0], np.float32), size=n)
    for k in sorted({0, 1, n // 3, n // 2, n - 1, n} - {-1}):
        if k < 0:
            continue
        got = O.select_topk(vals, k, 1000)
        assert got.tolist() == _brute_select(vals.tolist(), k, 1000)


def test_select_edge_cases():
    eq = np.full(10, 7.0, np.float32)
    assert O.select_topk(eq, 3, 5).tolist() == [5, 6, 7]          # equal scores: lowest indices
    assert O.select_topk(eq, 0).tolist() == []
    assert O.select_topk(eq, 10).tolist() == list(range(10))
    special = np.array([1.0, np.inf, np.nan, 0.0, -1.0, 3.0], np.float32)
    # +NaN ranks above +inf, +inf above every finite value, negatives lowest
    assert O.select_topk(special, 1).tolist() == [2]
    assert O.select_topk(special, 2).tolist() == [1, 2]
    assert O.select_topk(special, 3).tolist() == [1, 2, 5]
    assert O.select_topk(special, 5).tolist() == [0, 1, 2, 3, 5]
    with pytest.raises(ValueError):
        O.select_topk(eq, 11)


def test_k_from_rho_and_cache_fraction(golden):
    rf = golden["repair_fraction"]
    C = 1024
    n_cand = (rf["chunks"] - 1) * C
    k = O.k_from_rho(int(round(rf["rho"] * 10000)), n_cand)
    assert k == 1076                              # ceil(0.35 * 3072) = ceil(1075.2)
    assert abs(k / (rf["chunks"] * C) - rf["composed_cache_fraction_approx"]) < 0.02
    assert O.k_from_rho(1500, 63488) == 9524      # ceil(9523.2)
    assert O.k_from_rho(1500, 3072) == 461
    assert O.k_from_rho(0, 5) == 0 and O.k_from_rho(10000, 5) == 5


# ---------------------------------------------------------- attention ----

def _sdpa_reference(q, k, v, qpos, scale):
    """torch SDPA (CPU, fp64) with an explicit boolean mask and repeated kv heads."""
    L, M, Hq, Dd = q.shape
    T, Hkv = k.shape[1], k.shape[2]
    G = Hq // Hkv
    out = np.zeros(q.shape)
    mask = torch.from_numpy(np.arange(T)[None, :] <= np.asarray(qpos)[:, None])   # [M, T]
    for l in range(L):
        qq = torch.from_numpy(q[l]).permute(1, 0, 2)                             # [Hq, M, D]
        kk = torch.from_numpy(k[l]).permute(1, 0, 2).repeat_interleave(G, dim=0)  # [Hq, T, D]
        vv = torch.from_numpy(v[l]).permute(1, 0, 2).repeat_interleave(G, dim=0)
        o = torch.nn.functional.scaled_dot_product_attention(qq, kk, vv, attn_mask=mask,
                                                             scale=scale)
        out[l] = o.permute(1, 0, 2).numpy()
    return out


@pytest.mark.parametrize("Hq,Hkv", [(2, 1), (16, 2), (28, 4), (4, 4)])
def test_attention_matches_torch_sdpa(Hq, Hkv):
    rng = np.random.default_rng(Hq * 10 + Hkv)
    L, T, M, Dd = 2, 40, 9, 128
    q = rng.standard_normal((L, M, Hq, Dd))
    k = rng.standard_normal((L, T, Hkv, Dd))
    v = rng.standard_normal((L, T, Hkv, Dd))
    qpos = np.sort(rng.choice(T, size=M, replace=False))
    o, lse = O.repair_attention(q, k, v, qpos)
    ref = _sdpa_reference(q, k, v, qpos, 1.0 / math.sqrt(Dd))
    np.testing.assert_allclose(o, ref, atol=1e-12)
    # the normaliser: logsumexp of the visible scaled logits
    l, r, h = 1, M - 1, Hq - 1
    s = torch.from_numpy(k[l, :qpos[r] + 1, h // (Hq // Hkv)] @ q[l, r, h] / math.sqrt(Dd))
    assert lse[l, r, h] == pytest.approx(float(torch.logsumexp(s, 0)), abs=1e-12)


def test_attention_special_cases():
    rng = np.random.default_rng(11)
    L, T, Hq, Hkv = 1, 20, 4, 2
    q = rng.standard_normal((L, 3, Hq, D))
    k = rng.standard_normal((L, T, Hkv, D))
    v = rng.standard_normal((L, T, Hkv, D))
    qpos = np.array([0, 5, 19])
    o, _ = O.repair_attention(q, k, v, qpos)
    # one visible key: the output is that key's value
    np.testing.assert_allclose(o[0, 0, 0], v[0, 0, 0], atol=1e-15)
    np.testing.assert_allclose(o[0, 0, 3], v[0, 0, 1], atol=1e-15)
    # zero query: uniform weights, the mean of the visible values
    o0, _ = O.repair_attention(np.zeros_like(q), k, v, qpos)
    np.testing.assert_allclose(o0[0, 1, 2], v[0, :6, 1].mean(axis=0), atol=1e-14)
    np.testing.assert_allclose(o0[0, 2, 1], v[0, :20, 0].mean(axis=0), atol=1e-14)


def test_attention_all_rows_is_full_causal_attention():
    rng = np.random.default_rng(12)
    L, T, Hq, Hkv = 1, 24, 2, 1
    x = rng.standard_normal((L, T, Hq, D))
    k = rng.standard_normal((L, T, Hkv, D))
    v = rng.standard_normal((L, T, Hkv, D))
    o, _ = O.repair_attention(x, k, v, np.arange(T))
    s = np.einsum("thd,jd->thj", x[0], k[0, :, 0]) / math.sqrt(D)
    s = np.where(np.arange(T)[None, None, :] <= np.arange(T)[:, None, None], s, -np.inf)
    p = np.exp(s - s.max(-1, keepdims=True))
    p /= p.sum(-1, keepdims=True)
    np.testing.assert_allclose(o[0], np.einsum("thj,jd->thd", p, v[0, :, 0]), atol=1e-13)


def test_attention_invariant_under_common_shift():
    rng = np.random.default_rng(13)
    T, Hq, Hkv = 30, 4, 2
    k = rng.standard_normal((1, T, Hkv, D))
    v = rng.standard_normal((1, T, Hkv, D))
    qrows = np.array([3, 10, 29])
    q = rng.standard_normal((1, 3, Hq, D))
    p = rng.integers(0, 100, size=(T, 3))
    o1, _ = O.repair_attention(q, k, v, qrows)
    shift = np.array([[64, 64, 64]])
    ks = O.rebase_f64(k, p, p + shift)
    qs = O.rebase_f64(q, p[qrows], p[qrows] + shift)
    o2, _ = O.repair_attention(qs, ks, v, qrows)
    np.testing.assert_allclose(o2, o1, atol=1e-11)


def test_scatter_rows_by_definition():
    """Scatter-back (Sec. 2): a hand-built case, the identity when the rows already are the
    cache's, and every untouched row bit-identical."""
    cache = np.arange(2 * 5 * 3, dtype=np.float64).reshape(2, 5, 3)
    rows = -np.arange(1, 2 * 2 * 3 + 1, dtype=np.float64).reshape(2, 2, 3)
    out = O.scatter_rows(cache, rows, [3, 0])
    exp = cache.copy()
    exp[0, 3], exp[1, 3] = [-1, -2, -3], [-7, -8, -9]
    exp[0, 0], exp[1, 0] = [-4, -5, -6], [-10, -11, -12]
    assert np.array_equal(out, exp)
    assert np.array_equal(cache, np.arange(30, dtype=np.float64).reshape(2, 5, 3))   # input kept
    rng = np.random.default_rng(3)
    big = rng.standard_normal((3, 40, 2, 8))
    idx = np.sort(rng.choice(40, 11, replace=False))
    assert np.array_equal(O.scatter_rows(big, big[:, idx], idx), big)
    fresh = rng.standard_normal((3, 11, 2, 8))
    got = O.scatter_rows(big, fresh, idx)
    keep = np.setdiff1d(np.arange(40), idx)
    assert np.array_equal(got[:, keep], big[:, keep]) and np.array_equal(got[:, idx], fresh)
