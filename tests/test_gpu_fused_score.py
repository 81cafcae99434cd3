"""cs_rebase_and_score (steps 1 and 2 in one launch) against the two separate calls on the
same inputs: re-based keys and scores must agree bit for bit, for every kv head count and
both storage types (the fused score reduces a token's block sums by lane shuffles when its
row fits one warp, through shared memory otherwise, and from registers in the fp32
kernel); and against the oracle's canonical score."""
import numpy as np
import pytest
import torch

import cs_workloads as W
import oracle as O
from _helpers import bits16, cuda, f64

pytestmark = pytest.mark.gpu


def _inputs(L, T, H, dtype, seed, n_cand, cand0, sl=1):
    g = torch.Generator().manual_seed(seed)
    k = torch.randn(L, T, H, 128, generator=g).to(dtype)
    fresh = (k[min(sl, L - 1), cand0:cand0 + n_cand].float() +
             0.3 * torch.randn(n_cand, H, 128, generator=g)).to(dtype)
    loc, glo = W.random_coordinates(T, seed)
    # a third of the tokens do not move (delta 0): their scores are still due
    still = np.random.default_rng(seed).random(T) < 0.33
    glo[still] = loc[still]
    return k, fresh, loc, glo


@pytest.mark.parametrize("H,dtype,in_place,L,sl", [
    (1, torch.bfloat16, True, 3, 1), (2, torch.bfloat16, True, 3, 1),
    (4, torch.bfloat16, False, 3, 1), (8, torch.bfloat16, True, 3, 1),
    (8, torch.bfloat16, False, 6, 5), (3, torch.bfloat16, True, 3, 1),
    (7, torch.bfloat16, False, 3, 2), (16, torch.bfloat16, True, 2, 1),
    (1, torch.float32, True, 3, 1), (2, torch.float32, True, 3, 1),
    (2, torch.float32, False, 6, 5), (3, torch.float32, True, 5, 4),
    (8, torch.float32, False, 3, 0), (16, torch.float32, True, 2, 1)])
def test_fused_equals_separate_calls(cslib, H, dtype, in_place, L, sl):
    T, cand0, n_cand = 203, 17, 161
    k, fresh, loc, glo = _inputs(L, T, H, dtype, 40 + H, n_cand, cand0, sl)
    pl, pg = cuda(loc), cuda(glo)
    # separate calls
    kb = k.cuda()
    cslib.cs_rebase_keys(kb, pl, pg)
    s_sep = cslib.cs_score_deviation(fresh.cuda(), kb[sl, cand0:cand0 + n_cand])
    # one call
    ka = k.cuda()
    out = None if in_place else torch.full_like(ka, float("nan"))
    res, s_one = cslib.cs_rebase_and_score(ka, pl, pg, fresh.cuda(), sl, cand0, k_out=out)
    cslib.cs_sync_status()
    if not in_place:
        assert np.array_equal(f64(ka), f64(k))          # input untouched
    if dtype == torch.bfloat16:
        assert np.array_equal(bits16(res), bits16(kb))
    else:
        assert np.array_equal(f64(res), f64(kb))
    assert np.array_equal(s_one.cpu().numpy().view(np.uint32), s_sep.cpu().numpy().view(np.uint32))


@pytest.mark.parametrize("H", [2, 4, 8, 16])
def test_fused_score_matches_oracle(cslib, H):
    L, T, cand0, n_cand = 2, 140, 40, 100
    k, fresh, loc, glo = _inputs(L, T, H, torch.bfloat16, 70 + H, n_cand, cand0)
    exp_k, _ = O.rebase(f64(k[1])[None], loc, glo, "bf16")
    exp = O.score_f32_canonical(f64(fresh).astype(np.float32),
                                exp_k[0, cand0:cand0 + n_cand].astype(np.float32))
    _, got = cslib.cs_rebase_and_score(k.cuda(), cuda(loc), cuda(glo), fresh.cuda(), 1, cand0)
    cslib.cs_sync_status()
    assert np.array_equal(got.cpu().numpy().view(np.uint32), exp.view(np.uint32))


@pytest.mark.parametrize("H", [1, 2, 5])
def test_fused_score_f32_matches_oracle(cslib, H):
    """fp32 storage: the re-base is within a few ulps of the oracle (not bit for bit), so the
    score is checked stage-wise: the oracle's canonical score of the keys the GPU re-based,
    bit for bit, and the keys within the fp32 tolerance of the oracle's rotation."""
    L, T, cand0, n_cand = 3, 150, 30, 120
    k, fresh, loc, glo = _inputs(L, T, H, torch.float32, 90 + H, n_cand, cand0)
    exp_k, _ = O.rebase(f64(k[1])[None], loc, glo, "f32")
    res, got = cslib.cs_rebase_and_score(k.cuda(), cuda(loc), cuda(glo), fresh.cuda(), 1, cand0)
    cslib.cs_sync_status()
    assert np.max(np.abs(f64(res[1]) - exp_k[0])) <= 1e-5
    exp = O.score_f32_canonical(f64(fresh).astype(np.float32),
                                f64(res[1, cand0:cand0 + n_cand]).astype(np.float32))
    assert np.array_equal(got.cpu().numpy().view(np.uint32), exp.view(np.uint32))


def test_fused_edge_cases(cslib):
    L, T, H = 2, 64, 2
    k, fresh, loc, glo = _inputs(L, T, H, torch.bfloat16, 5, 64, 0)
    # no candidates: a plain re-base
    kb = k.cuda()
    cslib.cs_rebase_keys(kb, cuda(loc), cuda(glo))
    res, s = cslib.cs_rebase_and_score(k.cuda(), cuda(loc), cuda(glo), fresh[:0].cuda(), 0, 10)
    cslib.cs_sync_status()
    assert s.numel() == 0 and np.array_equal(bits16(res), bits16(kb))
    # every token a candidate, score layer 0, the last candidate at T-1
    _, s_all = cslib.cs_rebase_and_score(k.cuda(), cuda(loc), cuda(glo), fresh.cuda(), 0, 0)
    s_ref = cslib.cs_score_deviation(fresh.cuda(), kb[0])
    cslib.cs_sync_status()
    assert np.array_equal(s_all.cpu().numpy().view(np.uint32), s_ref.cpu().numpy().view(np.uint32))
    with pytest.raises(cslib.CsError):
        cslib.cs_rebase_and_score(k.cuda(), cuda(loc), cuda(glo), fresh[:10].cuda(), 2, 0)   # layer 2 of 2
    with pytest.raises(cslib.CsError):
        cslib.cs_rebase_and_score(k.cuda(), cuda(loc), cuda(glo), fresh[:10].cuda(), 0, 60)  # past T
