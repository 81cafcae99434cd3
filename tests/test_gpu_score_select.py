"""Score (Eq. 5) and top-rho selection (Sec. 2) on the GPU against the oracle.

The score that the selection ranks is defined in one fixed fp32 order, so GPU
and oracle must agree bit for bit; indices must agree exactly."""
import numpy as np
import pytest
import torch

import oracle as O
from _helpers import cuda, f64

pytestmark = pytest.mark.gpu


def _rows(n, H, dtype, seed, scale=1.0):
    g = torch.Generator(device="cuda").manual_seed(seed)
    return (torch.randn((n, H, 128), generator=g, device="cuda") * scale).to(dtype)


@pytest.mark.parametrize("H", [1, 2, 4, 7, 8, 16])
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("n", [1, 37, 3072])
def test_score_bit_exact(cslib, H, dtype, n):
    a = _rows(n, H, dtype, 1 + H + n)
    b = (a.float() + _rows(n, H, torch.float32, 7 + H + n) *
         torch.exp(_rows(n, 1, torch.float32, 9)[:, :, :1])).to(dtype)
    got = cslib.cs_score_deviation(a, b)
    cslib.cs_sync_status()
    exp = O.score_f32_canonical(f64(a).astype(np.float32), f64(b).astype(np.float32))
    assert np.array_equal(got.cpu().numpy().view(np.uint32), exp.view(np.uint32))
    np.testing.assert_allclose(got.cpu().numpy(), O.score_f64(f64(a), f64(b)), rtol=2e-6)


def test_score_strided_rows_and_exact_cases(cslib):
    # rows taken from a [L, T, H, D] cache slice: stride H*D, plus a padded fresh buffer
    cache = _rows(4 * 50, 2, torch.bfloat16, 3).view(4, 50, 2, 128)
    cached = cache[1, 10:40]
    fresh_buf = torch.zeros((30, 3, 128), dtype=torch.bfloat16, device="cuda")
    fresh_buf[:, :2] = _rows(30, 2, torch.bfloat16, 4)
    fresh = fresh_buf[:, :2]
    got = cslib.cs_score_deviation(fresh, cached)
    cslib.cs_sync_status()
    exp = O.score_f32_canonical(f64(fresh).astype(np.float32), f64(cached).astype(np.float32))
    assert np.array_equal(got.cpu().numpy().view(np.uint32), exp.view(np.uint32))
    same = cslib.cs_score_deviation(cached.contiguous(), cached)
    cslib.cs_sync_status()
    assert torch.count_nonzero(same).item() == 0
    # worked by hand: ((1 + 2^-24) + (2^-24 + 2^-24)) = 1 + 2^-23 in the fixed order
    a = torch.zeros((1, 2, 128), dtype=torch.float32, device="cuda")
    a[0, 0, :4] = torch.tensor([1.0, 2 ** -12, 2 ** -12, 2 ** -12])
    z = cslib.cs_score_deviation(a, torch.zeros_like(a))
    cslib.cs_sync_status()
    assert z.item() == np.float32(1.0 + 2.0 ** -23)


def _check_select(cs, vals, k, base):
    s = cuda(np.asarray(vals, np.float32))
    got = cs.cs_select_topk(s, k, base)
    cs.cs_sync_status()
    exp = O.select_topk(np.asarray(vals, np.float32), k, base)
    assert np.array_equal(got.cpu().numpy(), exp)


# n spans every cluster size of the select (1, 2, 4, 8, 16 CTAs), the keys-in-registers
# variants (4, 8, 16 per thread) and the re-read variant (n > 131072), with ragged tails
@pytest.mark.parametrize("n", [1, 7, 1023, 1024, 1025, 3072, 4096, 4097, 8191, 8193, 15360, 16384,
                               16385, 32769, 64512, 100003, 131073, 262147])
def test_select_matches_oracle(cslib, n):
    rng = np.random.default_rng(n)
    cont = (rng.lognormal(0, 1.5, n) * 256).astype(np.float32)
    ties = rng.choice(np.array([0, 1, 2, 3.5, 1e30], np.float32), n)
    for vals in (cont, ties):
        for k in sorted({0, 1, n // 7, n // 2, max(n - 1, 0), n}):
            _check_select(cslib, vals, k, 1032)


def test_select_special_values(cslib):
    vals = np.array([1.0, np.inf, np.nan, 0.0, -1.0, 3.0, -0.0, -np.inf, 3.0, np.inf],
                    np.float32)
    for k in range(len(vals) + 1):
        _check_select(cslib, vals, k, 0)
    eq = np.full(5000, 2.5, np.float32)
    _check_select(cslib, eq, 1234, 17)        # all equal: lowest indices


def test_select_fraction_of_candidates(cslib):
    """k = ceil(rho * N_c) of the candidates with idx_base at the first candidate."""
    rng = np.random.default_rng(0)
    n_cand, cand0 = 3072, 1032
    vals = (rng.lognormal(0, 1, n_cand) * 256).astype(np.float32)
    k = O.k_from_rho(1500, n_cand)
    s = cuda(vals)
    got = cslib.cs_select_topk(s, k, cand0).cpu().numpy()
    cslib.cs_sync_status()
    assert len(got) == 461 and got[0] >= cand0 and got[-1] < cand0 + n_cand
    assert np.all(np.diff(got) > 0)
    kth = np.sort(vals)[::-1][k - 1]
    assert np.all(vals[got - cand0] >= kth)


@pytest.mark.parametrize("n", [5000, 70001])
def test_select_unaligned_scores(cslib, n):
    """Scores that start 4 bytes past a 16-byte boundary take the scalar-load path."""
    rng = np.random.default_rng(n + 1)
    vals = (rng.lognormal(0, 1.5, n + 1) * 256).astype(np.float32)
    buf = cuda(vals)
    view = buf[1:]
    assert view.data_ptr() % 16 == 4
    for k in (1, n // 3, n - 1):
        got = cslib.cs_select_topk(view, k, 9).cpu().numpy()
        cslib.cs_sync_status()
        assert np.array_equal(got, O.select_topk(vals[1:], k, 9))


def test_select_ties_across_ctas(cslib):
    """All scores equal over 64 512 candidates (16 CTAs): the k lowest indices, so every
    CTA's share of the ties depends on the CTAs before it."""
    n = 64512
    vals = np.full(n, 7.25, np.float32)
    vals[::1000] = 9.0
    for k in (1, 65, 30000, n - 3):
        _check_select(cslib, vals, k, 1032)


@pytest.mark.parametrize("n", [2, 100, 3000, 4096, 6000, 8192])
def test_select_small_input_paths(cslib, n):
    """Inputs of one CTA (up to 8 192 scores): a key range spanning all 32 bits, a tight
    cluster that needs three digit passes (the keys differ only in their 12 lowest bits
    below two outliers), a range of a few low bits only, signed values, and scores that
    start 4 bytes past a 16-byte boundary."""
    rng = np.random.default_rng(7 * n)
    wide = (rng.lognormal(0, 3, n) * rng.choice([-1.0, 1.0], n)).astype(np.float32)
    bits = (np.float32(1.0).view(np.uint32) + rng.integers(0, 4096, n)).astype(np.uint32)
    cluster = bits.view(np.float32).copy()
    cluster[0], cluster[-1] = 1e30, 0.0
    narrow = (np.float32(3.0).view(np.uint32) + rng.integers(0, 8, n)).astype(np.uint32)
    narrow = narrow.view(np.float32)
    for vals in (wide, cluster, narrow):
        for k in sorted({1, max(n // 10, 1), n // 2, max(n - 1, 1)}):
            _check_select(cslib, vals, k, 5)
    buf = cuda(np.concatenate([[np.float32(9.0)], wide]).astype(np.float32))
    view = buf[1:]
    assert view.data_ptr() % 16 == 4
    for k in sorted({1, max(n // 3, 1), max(n - 1, 1)}):
        got = cslib.cs_select_topk(view, k, 0).cpu().numpy()
        cslib.cs_sync_status()
        assert np.array_equal(got, O.select_topk(wide, k, 0))
