"""Repair attention (Eq. 1 over selected rows, causal in global order) on the GPU
against the fp64 oracle: max-abs 2e-2 for bf16 outputs, 1e-5 for fp32."""
import numpy as np
import pytest
import torch

import cs_workloads as W
import oracle as O
from _helpers import TOL, cuda, f64

pytestmark = pytest.mark.gpu


def _rand(shape, seed, dtype):
    g = torch.Generator(device="cuda").manual_seed(seed)
    return torch.randn(shape, generator=g, device="cuda").to(dtype)


def _run_and_check(cs, q, k, v, qpos, name, rows=None, layers=None, check_lse=True):
    L, M, Hq, D = q.shape
    lse = torch.full((L, M, Hq), float("nan"), dtype=torch.float32, device="cuda")
    out = cs.cs_repair_attention(q, k, v, cuda(qpos), lse=lse)
    cs.cs_sync_status()
    rows = np.arange(M) if rows is None else np.asarray(rows)
    layers = np.arange(L) if layers is None else np.asarray(layers)
    qq = f64(q[torch.as_tensor(layers, device="cuda")][:, torch.as_tensor(rows, device="cuda")])
    kk = f64(k[torch.as_tensor(layers, device="cuda")])
    vv = f64(v[torch.as_tensor(layers, device="cuda")])
    eo, el = O.repair_attention(qq, kk, vv, np.asarray(qpos)[rows])
    go = f64(out[torch.as_tensor(layers, device="cuda")][:, torch.as_tensor(rows, device="cuda")])
    err = np.max(np.abs(go - eo))
    assert err <= TOL[name], f"max abs error {err}"
    if check_lse:
        gl = lse[torch.as_tensor(layers, device="cuda")][:, torch.as_tensor(rows, device="cuda")]
        np.testing.assert_allclose(gl.cpu().numpy(), el, atol=1e-3 if name == "bf16" else 1e-5)
    return err


def test_tiny_f32_config_full(cslib):
    w = W.CONFIGS["tiny_f32"]
    x = W.make_inputs(w, seed=0, device="cuda")
    rng = np.random.default_rng(0)
    qpos = np.sort(rng.choice(np.arange(w.cand0, w.T), size=w.M, replace=False)).astype(np.int32)
    _run_and_check(cslib, x["q"], x["k"], x["v"], qpos, "f32")


@pytest.mark.parametrize("Hq,Hkv", [(2, 1), (8, 2), (6, 3)])
def test_f32_key_chunks_ragged(cslib, Hq, Hkv):
    """fp32 path: rows whose visible keys end on, before and after the 32-key chunk edges,
    including the first key alone, over two layers."""
    L, T = 2, 300
    qpos = np.array([0, 1, 30, 31, 32, 33, 63, 64, 65, 100, 127, 128, 200, 299], np.int32)
    M = len(qpos)
    q = _rand((L, M, Hq, 128), 21, torch.float32)
    k = _rand((L, T, Hkv, 128), 22, torch.float32)
    v = _rand((L, T, Hkv, 128), 23, torch.float32)
    _run_and_check(cslib, q, k, v, qpos, "f32")


@pytest.mark.parametrize("Hq,Hkv", [(16, 2), (28, 4), (2, 1), (8, 8), (7, 1), (32, 2)])
def test_bf16_group_sizes_ragged(cslib, Hq, Hkv):
    L, T, M = 2, 1000, 37
    q = _rand((L, M, Hq, 128), 1, torch.bfloat16)
    k = _rand((L, T, Hkv, 128), 2, torch.bfloat16)
    v = _rand((L, T, Hkv, 128), 3, torch.bfloat16)
    rng = np.random.default_rng(Hq)
    qpos = np.sort(rng.choice(T, size=M, replace=False)).astype(np.int32)
    qpos[0] = 0
    _run_and_check(cslib, q, k, v, qpos, "bf16")


@pytest.mark.parametrize("seed", range(6))
def test_bf16_random_shapes(cslib, seed):
    """Seeded random shapes: GQA groups that do not divide 128 (3, 5, 6: tiles of 126, 125 and
    126 rows with spare rows zeroed), ragged key counts, several layers, random positions."""
    rng = np.random.default_rng(100 + seed)
    G = [3, 5, 6, 12, 4, 1][seed]
    Hkv = int(rng.choice([1, 2, 3]))
    L = int(rng.integers(1, 4))
    T = int(rng.integers(130, 900))
    M = int(rng.integers(1, min(T, 90)))
    q = _rand((L, M, G * Hkv, 128), 200 + seed, torch.bfloat16)
    k = _rand((L, T, Hkv, 128), 300 + seed, torch.bfloat16)
    v = _rand((L, T, Hkv, 128), 400 + seed, torch.bfloat16)
    qpos = np.sort(rng.choice(T, size=M, replace=False)).astype(np.int32)
    _run_and_check(cslib, q, k, v, qpos, "bf16")


def test_bf16_dense_rows_and_block_edges(cslib):
    """Consecutive rows and rows on key-block boundaries (127, 128, 255, 256, ...)."""
    L, T, Hq, Hkv = 1, 700, 16, 2
    q = _rand((L, 40, Hq, 128), 4, torch.bfloat16)
    k = _rand((L, T, Hkv, 128), 5, torch.bfloat16)
    v = _rand((L, T, Hkv, 128), 6, torch.bfloat16)
    qpos = np.array(sorted(set(list(range(0, 20)) + [126, 127, 128, 129, 254, 255, 256, 257,
                                                        383, 384, 511, 512, 513, 639, 640,
                                                        698, 699])), np.int32)[:40]
    q = q[:, :len(qpos)].contiguous()
    _run_and_check(cslib, q, k, v, qpos, "bf16")


def test_bf16_large_logits_rescale(cslib):
    """Keys growing along the sequence force the running maximum to rise block after block."""
    L, T, Hq, Hkv = 1, 1024, 8, 1
    q = _rand((L, 16, Hq, 128), 7, torch.float32)
    k = _rand((L, T, Hkv, 128), 8, torch.float32) * torch.linspace(0.1, 4.0, T,
                                                                   device="cuda")[None, :, None, None]
    v = _rand((L, T, Hkv, 128), 9, torch.float32)
    qpos = np.linspace(100, T - 1, 16).astype(np.int32)
    _run_and_check(cslib, (q * 2).to(torch.bfloat16), k.to(torch.bfloat16),
                   v.to(torch.bfloat16), qpos, "bf16")


def test_bf16_max_grows_in_one_half(cslib):
    """One large key in the first half of block 1's columns, a larger one in the second half of
    block 2's: the running maximum of the rows that see them rises by more than 2^8 in one
    64-column half only, so both halves of those rows must take the new maximum together."""
    L, T, Hq, Hkv = 1, 512, 8, 1
    q = torch.full((L, 16, Hq, 128), 0.5, device="cuda")
    k = _rand((L, T, Hkv, 128), 15, torch.float32) * 0.1
    v = _rand((L, T, Hkv, 128), 16, torch.float32)
    k[0, 150] = 1.5          # block 1, column 22: scores +8.5 (x log2(e) > 8)
    k[0, 330] = 3.0          # block 2, column 74: scores +17
    qpos = np.array([100, 149, 150, 151, 200, 255, 256, 300, 329, 330, 331, 383, 384, 400,
                     450, 511], np.int32)
    _run_and_check(cslib, q.to(torch.bfloat16), k.to(torch.bfloat16), v.to(torch.bfloat16),
                   qpos, "bf16")


def test_bf16_growth_flag_thresholds(cslib):
    """The regimes of the softmax's growth check (a block is flagged when its weights, taken with
    the running maximum of the earlier blocks, sum above 2^12): one key about 2^10 above the
    running maximum (not flagged: weights up to 2^10 stay in the running sum), then 64 keys of
    one half block about 2^6.3 above it (flagged by their sum, while the maximum grows by less
    than the 2^8 at which the running maximum is raised).  A constant query q = 0.5 against a
    constant key c gives a log2-domain score of 0.5 * c * 128 / sqrt(128) * log2(e) = 8.16 c."""
    L, T, Hq, Hkv = 1, 512, 8, 1
    q = torch.full((L, 16, Hq, 128), 0.5, device="cuda")
    k = _rand((L, T, Hkv, 128), 17, torch.float32) * 0.1
    v = _rand((L, T, Hkv, 128), 18, torch.float32)
    k[0, 150] = 10.0 / 8.16          # block 1, column 22: about 2^10 above block 0's maximum
    k[0, 320:384] = 6.5 / 8.16       # block 2, columns 64-127: 64 weights of about 2^6.3
    qpos = np.array([100, 149, 150, 151, 200, 255, 256, 300, 319, 320, 321, 350, 383, 384,
                     450, 511], np.int32)
    _run_and_check(cslib, q.to(torch.bfloat16), k.to(torch.bfloat16), v.to(torch.bfloat16),
                   qpos, "bf16")


def test_qwen3b_4x1024_all_rows(cslib):
    w = W.CONFIGS["qwen3b_4x1024"]
    x = W.make_inputs(w, seed=0, device="cuda")
    rng = np.random.default_rng(1)
    qpos = np.sort(rng.choice(np.arange(w.cand0, w.cand0 + w.n_cand), size=w.M,
                              replace=False)).astype(np.int32)
    _run_and_check(cslib, x["q"], x["k"], x["v"], qpos, "bf16", layers=[0, 1, 17, 35])


@pytest.mark.parametrize("name", ["qwen3b_16x1024_q64", "qwen3b_64x1024_r30", "qwen7b_32x2048"])
def test_large_configs_sampled_rows(cslib, name):
    w = W.CONFIGS[name]
    x = W.make_inputs(w, seed=0, device="cuda")
    rng = np.random.default_rng(2)
    sel = np.sort(rng.choice(np.arange(w.cand0, w.cand0 + w.n_cand), size=w.k, replace=False))
    qpos = np.concatenate([sel, np.arange(w.T - w.suffix, w.T)]).astype(np.int32)
    rows = W.sample_rows(w.M, 48, seed=5)
    _run_and_check(cslib, x["q"], x["k"], x["v"], qpos, "bf16", rows=rows,
                   layers=[0, w.n_layers - 1])


def test_single_key_and_empty(cslib):
    q = _rand((1, 1, 16, 128), 10, torch.bfloat16)
    k = _rand((1, 5, 2, 128), 11, torch.bfloat16)
    v = _rand((1, 5, 2, 128), 12, torch.bfloat16)
    out = cslib.cs_repair_attention(q, k, v, cuda(np.array([0], np.int32)))
    cslib.cs_sync_status()
    # one visible key: every head of group g returns v[0, 0, g]
    for h in range(16):
        assert torch.allclose(out[0, 0, h].float(), v[0, 0, h // 8].float(), atol=1e-2)
    empty = cslib.cs_repair_attention(q[:, :0].contiguous(), k, v,
                                      cuda(np.zeros(0, np.int32)))
    cslib.cs_sync_status()
    assert empty.numel() == 0


def test_binding_rejects_a_head_dim_mismatch(cslib):
    """K and V must have Q's head dim: with one layer no stride would give the mismatch away."""
    q = _rand((1, 4, 16, 128), 17, torch.bfloat16)
    k = _rand((1, 64, 2, 64), 18, torch.bfloat16)
    with pytest.raises(ValueError):
        cslib.cs_repair_attention(q, k, k, cuda(np.array([3, 10, 20, 30], np.int32)))


def test_bad_query_positions_are_reported(cslib):
    q = _rand((1, 4, 16, 128), 13, torch.bfloat16)
    k = _rand((1, 64, 2, 128), 14, torch.bfloat16)
    bad = cuda(np.array([3, 10, 70, 20], np.int32))       # out of range and not ascending
    cslib.cs_repair_attention(q, k, k, bad)
    with pytest.raises(cslib.CsError) as e:
        cslib.cs_sync_status()
    assert e.value.status == cslib.CS_ERR_DEVICE_ARG
    cslib.cs_sync_status()                                 # cleared after reporting
    q32, k32 = q.float(), k.float()
    cslib.cs_repair_attention(q32, k32, k32, bad)
    with pytest.raises(cslib.CsError):
        cslib.cs_sync_status()
