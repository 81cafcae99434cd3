"""Synthetic, seeded ChronoStitch workloads: shapes, coordinates and random tensors.

This module is shared by the CPU oracle's tests and by the CUDA path's tests and
benchmark. It holds no arithmetic of the method (no rotation, no scoring, no
selection, no attention): only the workload shapes, the token-coordinate layout
and seeded random draws.

Workload structure (ChronoStitch, Sec. 2 and Sec. 3):
  * a composed sequence is   [text prefix P][chunk 0]...[chunk N-1][text suffix S]
    with C = grid_t * grid_h * grid_w visual tokens per chunk, raster order
    (t-major, then h, then w), T = P + N*C + S tokens in all;
  * each chunk was prefilled independently, so its stored keys carry local
    three-axis coordinates; composition moves them to a global,
    non-overlapping coordinate interval (Sec. 2, Eq. 3);
  * candidates for repair are the visual tokens of chunks 1..N-1 (the
    "later-chunk" tokens, Sec. 2), a contiguous global index range;
  * k = ceil(rho * N_c) of them are selected (Sec. 2, top-rho fraction).

Random tensors:
  * stored keys K [L, T, Hkv, D] ~ N(0, 1).  A stored key is f(x, p_local) for a
    pre-rotary key x (Eq. 2); f is orthogonal, so for x ~ N(0, I) the stored key
    is itself N(0, I): drawing it directly needs no rotation.
  * values V [L, T, Hkv, D] ~ N(0, 1); queries of the repaired rows
    Q [L, M, Hq, D] ~ N(0, 1) (post-rotary at global coordinates, same argument).
  * fresh keys: per candidate a scale s_t ~ LogNormal(0, sigma) and noise
    eps_t ~ N(0, I); the perturbed layer-1 stored key  K[1, t] + s_t * eps_t,
    rounded to the storage dtype, is returned in LOCAL coordinates.  The fresh
    key at global coordinates (what a shallow recompute would produce) is that
    tensor re-based by Eq. 3, which each side (oracle, CUDA path) computes with
    its own implementation.
"""
from __future__ import annotations

import dataclasses

import numpy as np
import torch

HEAD_DIM = 128
MROPE_SECTIONS = (16, 24, 24)   # temporal, height, width frequency pairs (Sec. 3)
ROPE_THETA = 1.0e6              # Qwen2.5-VL rotary base


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    n_layers: int
    n_chunks: int
    grid_t: int
    grid_h: int
    grid_w: int
    prefix: int
    suffix: int
    hq: int
    hkv: int
    rho_bp: int          # repair fraction rho in basis points (1500 = 15 %)
    dtype: str           # "f32" or "bf16": storage dtype of K, V, Q, O
    sigma: float = 1.0   # lognormal sigma of the per-token fresh-key deviation scale
    layout: str = "segment"   # "segment" or "single_video" (see coordinates())
    head_dim: int = HEAD_DIM
    theta: float = ROPE_THETA
    sections: tuple = MROPE_SECTIONS

    # ---- derived sizes -------------------------------------------------
    @property
    def chunk_tokens(self) -> int:
        return self.grid_t * self.grid_h * self.grid_w

    @property
    def T(self) -> int:
        return self.prefix + self.n_chunks * self.chunk_tokens + self.suffix

    @property
    def t_vis(self) -> int:
        return self.n_chunks * self.chunk_tokens

    @property
    def cand0(self) -> int:
        """Global index of the first later-chunk visual token."""
        return self.prefix + self.chunk_tokens

    @property
    def n_cand(self) -> int:
        return (self.n_chunks - 1) * self.chunk_tokens

    @property
    def k(self) -> int:
        """k = ceil(rho * N_c), exact integer arithmetic on basis points."""
        return (self.rho_bp * self.n_cand + 9999) // 10000

    @property
    def M(self) -> int:
        """Query rows of the repair attention: selected tokens plus the text suffix."""
        return self.k + self.suffix

    @property
    def group(self) -> int:
        return self.hq // self.hkv

    @property
    def score_layer(self) -> int:
        """Layer whose keys are scored (layer 1, Eq. 5); layer 0 for a one-layer cache."""
        return min(1, self.n_layers - 1)

    @property
    def torch_dtype(self):
        return torch.float32 if self.dtype == "f32" else torch.bfloat16

    @property
    def elem_bytes(self) -> int:
        return 4 if self.dtype == "f32" else 2

    def with_(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


# The five workloads: one tiny fp32 case and four Qwen2.5-VL-shaped bf16 cases.
CONFIGS = {
    "tiny_f32": Workload("tiny_f32", n_layers=1, n_chunks=2, grid_t=2, grid_h=4, grid_w=4,
                         prefix=0, suffix=0, hq=2, hkv=1, rho_bp=2500, dtype="f32",
                         layout="single_video"),
    "qwen3b_4x1024": Workload("qwen3b_4x1024", n_layers=36, n_chunks=4, grid_t=4, grid_h=16,
                              grid_w=16, prefix=8, suffix=0, hq=16, hkv=2, rho_bp=1500,
                              dtype="bf16"),
    "qwen3b_16x1024_q64": Workload("qwen3b_16x1024_q64", n_layers=36, n_chunks=16, grid_t=4,
                                   grid_h=16, grid_w=16, prefix=8, suffix=64, hq=16, hkv=2,
                                   rho_bp=1500, dtype="bf16"),
    "qwen3b_64x1024_r05": Workload("qwen3b_64x1024_r05", n_layers=36, n_chunks=64, grid_t=4,
                                   grid_h=16, grid_w=16, prefix=8, suffix=0, hq=16, hkv=2,
                                   rho_bp=500, dtype="bf16", sigma=1.5),
    "qwen3b_64x1024_r15": Workload("qwen3b_64x1024_r15", n_layers=36, n_chunks=64, grid_t=4,
                                   grid_h=16, grid_w=16, prefix=8, suffix=0, hq=16, hkv=2,
                                   rho_bp=1500, dtype="bf16", sigma=1.5),
    "qwen3b_64x1024_r30": Workload("qwen3b_64x1024_r30", n_layers=36, n_chunks=64, grid_t=4,
                                   grid_h=16, grid_w=16, prefix=8, suffix=0, hq=16, hkv=2,
                                   rho_bp=3000, dtype="bf16", sigma=1.5),
    "qwen7b_32x2048": Workload("qwen7b_32x2048", n_layers=28, n_chunks=32, grid_t=4, grid_h=16,
                               grid_w=32, prefix=8, suffix=0, hq=28, hkv=4, rho_bp=1500,
                               dtype="bf16"),
}

# The workload the throughput number is quoted on: the largest single-GPU configuration
# of the 3B shape (64 chunks x 1024 tokens, the middle of its rho sweep).
BENCH_WORKLOAD = "qwen3b_64x1024_r15"


def coordinates(w: Workload):
    """Local (as stored) and global (composed) three-axis coordinates, int32 [T, 3].

    Text tokens carry one scalar position repeated on the three axes.  A visual
    token at grid cell (t, h, w) of its chunk has local coordinate
    (P + t, P + h, P + w): every chunk was prefilled after the same P-token
    text prefix, starting its own positions there.  Global coordinates:
      * "segment": chunk c is its own visual segment placed after the previous
        one, so all three axes move by c * S with S = max(grid_t, grid_h, grid_w)
        (each chunk gets a non-overlapping interval on every axis);
      * "single_video": the chunks are consecutive temporal grids of one video,
        so only the temporal axis moves, by c * grid_t.
    Suffix text tokens start one past the largest global coordinate.
    """
    P, C = w.prefix, w.chunk_tokens
    T = w.T
    loc = np.zeros((T, 3), dtype=np.int64)
    glo = np.zeros((T, 3), dtype=np.int64)
    ar = np.arange(P, dtype=np.int64)
    loc[:P] = ar[:, None]
    glo[:P] = ar[:, None]
    tt, hh, ww = np.meshgrid(np.arange(w.grid_t), np.arange(w.grid_h), np.arange(w.grid_w),
                             indexing="ij")
    cell = np.stack([tt.ravel(), hh.ravel(), ww.ravel()], axis=1).astype(np.int64)  # [C, 3]
    span = max(w.grid_t, w.grid_h, w.grid_w)
    for c in range(w.n_chunks):
        sl = slice(P + c * C, P + (c + 1) * C)
        loc[sl] = P + cell
        if w.layout == "segment":
            glo[sl] = P + cell + c * span
        elif w.layout == "single_video":
            shift = np.array([c * w.grid_t, 0, 0], dtype=np.int64)
            glo[sl] = P + cell + shift
        else:
            raise ValueError(f"unknown layout {w.layout!r}")
    if w.suffix:
        s0 = int(glo[:P + w.n_chunks * C].max()) + 1 if P + w.n_chunks * C else 0
        ar = s0 + np.arange(w.suffix, dtype=np.int64)
        loc[T - w.suffix:] = ar[:, None]
        glo[T - w.suffix:] = ar[:, None]
    return loc.astype(np.int32), glo.astype(np.int32)


def seed_for(w: Workload, seed: int, tensor_id: int, layer: int = 0) -> int:
    """Seed of one drawn tensor (and, for per-layer tensors, of one of its layers)."""
    base = seed * 1000003 + sum(map(ord, w.name)) * 101 + tensor_id
    return (base * 1009 + layer) & 0x7FFFFFFF


def _randn(shape, seed, device):
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    return torch.randn(shape, generator=g, device=device, dtype=torch.float32)


def _per_layer(w: Workload, shape, seed: int, tensor_id: int, layers, device, dtype):
    """[len(layers), *shape] in `dtype`; layer l is drawn from its own seed, so any
    subset of layers can be materialised without drawing the others."""
    out = torch.empty((len(layers),) + tuple(shape), dtype=dtype, device=device)
    for i, l in enumerate(layers):
        out[i] = _randn(shape, seed_for(w, seed, tensor_id, l), device).to(dtype)
    return out


def make_inputs(w: Workload, seed: int = 0, device="cpu", layers=None):
    """Seeded synthetic inputs for one composition query.

    Returns a dict of tensors on `device`:
      k [L,T,Hkv,D], v [L,T,Hkv,D]   stored cache (storage dtype), keys at local coords
      q [L,M,Hq,D]                   queries of the repaired rows (storage dtype)
      k_fresh_local [Nc,Hkv,D]       perturbed layer-1 stored keys, local coords
      pos_local, pos_global [T,3]    int32 coordinates
    Every layer of k, v and q is drawn from its own seed.  `layers` (a list of layer
    indices) materialises only those layers, in that order (the leading dimension is
    then len(layers)); k_fresh_local is the same whichever layers are asked for.  The
    draws use torch's generator for `device`; the same (workload, seed, device)
    always gives the same tensors.
    """
    T, Hkv, Hq, D = w.T, w.hkv, w.hq, w.head_dim
    dt = w.torch_dtype
    layers = list(range(w.n_layers)) if layers is None else [int(l) for l in layers]
    k = _per_layer(w, (T, Hkv, D), seed, 1, layers, device, dt)
    v = _per_layer(w, (T, Hkv, D), seed, 2, layers, device, dt)
    q = _per_layer(w, (w.M, Hq, D), seed, 3, layers, device, dt)
    nc = w.n_cand
    scale = torch.exp(w.sigma * _randn((nc, 1, 1), seed_for(w, seed, 4), device))
    eps = _randn((nc, Hkv, D), seed_for(w, seed, 5), device)
    sl = w.score_layer
    k_sl = k[layers.index(sl)] if sl in layers else _per_layer(w, (T, Hkv, D), seed, 1, [sl],
                                                               device, dt)[0]
    base = k_sl[w.cand0:w.cand0 + nc].float()
    k_fresh_local = (base + scale * eps).to(dt)
    loc, glo = coordinates(w)
    return {
        "k": k, "v": v, "q": q, "k_fresh_local": k_fresh_local,
        "pos_local": torch.from_numpy(loc).to(device),
        "pos_global": torch.from_numpy(glo).to(device),
    }


def random_coordinates(T: int, seed: int, max_coord: int = 4096):
    """Arbitrary per-token local and global coordinates (int32 [T,3]) for edge-case tests."""
    rng = np.random.default_rng(seed)
    loc = rng.integers(0, max_coord, size=(T, 3), dtype=np.int64)
    glo = rng.integers(0, max_coord, size=(T, 3), dtype=np.int64)
    return loc.astype(np.int32), glo.astype(np.int32)


def sample_rows(M: int, n: int, seed: int):
    """A seeded sample of at most n query rows, always holding the first and last."""
    if M <= n:
        return np.arange(M)
    rng = np.random.default_rng(seed)
    mid = rng.choice(np.arange(1, M - 1), size=n - 2, replace=False)
    return np.unique(np.concatenate([[0, M - 1], mid]))


def attention_flops(w: Workload, qpos: np.ndarray) -> float:
    """Algorithmic FLOP of the repair attention: 4*D per (layer, q head, visible key)."""
    vis = float(np.sum(qpos.astype(np.float64) + 1.0))
    return 4.0 * w.head_dim * w.hq * w.n_layers * vis


def rebase_bytes(w: Workload) -> float:
    """Algorithmic bytes of the re-base: read + write of every key row whose delta is non-zero."""
    loc, glo = coordinates(w)
    moved = int(np.any(loc != glo, axis=1).sum())
    return 2.0 * moved * w.n_layers * w.hkv * w.head_dim * w.elem_bytes


def score_bytes(w: Workload) -> float:
    """Algorithmic bytes of the score: two key rows read and one fp32 written per candidate."""
    return w.n_cand * (2.0 * w.hkv * w.head_dim * w.elem_bytes + 4.0)


def rebase_score_bytes(w: Workload, fused: bool) -> float:
    """Algorithmic bytes of re-base + score.  Fused into one launch, the score reads the
    fresh rows and writes one fp32 per candidate from HBM, and reads the rows it has just
    re-based back from L2 (not counted); as two launches it also reads those rows again."""
    fresh = w.n_cand * (w.hkv * w.head_dim * w.elem_bytes + 4.0)
    return rebase_bytes(w) + (fresh if fused else score_bytes(w))


def k_from_rho(rho_bp: int, n_cand: int) -> int:
    return (rho_bp * n_cand + 9999) // 10000


__all__ = ["Workload", "CONFIGS", "BENCH_WORKLOAD", "coordinates", "make_inputs",
           "random_coordinates", "sample_rows", "attention_flops", "rebase_bytes",
           "score_bytes", "rebase_score_bytes", "k_from_rho", "HEAD_DIM", "MROPE_SECTIONS", "ROPE_THETA"]
