"""CPU oracle for the ChronoStitch KV-composition hot path.

TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check of the build entry
point and the CPU-baseline leg of the benchmark may import this module.  The
CUDA library never calls it, and nothing here calls the CUDA library.

Plain, slow numpy code, written from the paper (arxiv 2607.19547, ChronoStitch):
  * mrope_rotate        Eq. 2      f(x, p): three-axis multimodal RoPE
  * rebase              Eq. 3      R(Delta) f(x, p) = f(x, p'), keys only
  * scalar1d_targets    Sec. 2     the scalar re-index baseline the paper rejects
  * score_f64 / score_f32_canonical   Eq. 5   delta_t = ||k_fresh - k_stored||_2 (squared)
  * select_topk         Sec. 2     top-rho later-chunk tokens
  * repair_attention    Eq. 1, Sec. 2   causal attention of the selected rows
  * scatter_rows        Sec. 2     fresh rows of the repaired tokens written into the cache
Floating point is fp64, with two deliberate exceptions where a float decides
an integer and both sides must take that decision in the same precision:
  * stored results are rounded to the storage dtype (round_to_bf16 / fp32 RN);
  * the score that the selection ranks is computed in fp32 in one fixed
    summation order (score_f32_canonical).
Readings of points the paper leaves open (theta schedule, pair layout, axis
order, tie-break, k from rho, causal order) are stated at each function.

Parity status: every function here is pinned by tests/test_oracle_pins.py
against closed forms, library routines (math.cos, torch SDPA, torch's bf16
conversion), brute force and the paper's printed figures.
"""
from __future__ import annotations

import numpy as np

# ----------------------------------------------------------------------------
# Eq. 2: three-axis mRoPE
# ----------------------------------------------------------------------------


def rope_theta(base: float, head_dim: int) -> np.ndarray:
    """theta_i = base^(-2i/D), i = 0..D/2-1 (the RoFormer schedule the paper cites).

    The paper writes theta_i without a formula (Eq. 2); this is the standard
    schedule of the RoPE it cites, with base 1e6 for Qwen2.5-VL.
    """
    i = np.arange(head_dim // 2, dtype=np.float64)
    return np.power(np.float64(base), -(2.0 * i) / head_dim)


def axis_of_pair(sections) -> np.ndarray:
    """sigma(i): the axis (0 = t, 1 = h, 2 = w) that frequency pair i follows.

    Sec. 3 gives 16 temporal, 24 height and 24 width frequencies; pairs are
    assigned to the axes in that order: [0,16) -> t, [16,40) -> h, [40,64) -> w.
    """
    return np.concatenate([np.full(int(n), a, dtype=np.int64) for a, n in enumerate(sections)])


def _rotate_pairs(x: np.ndarray, angle: np.ndarray) -> np.ndarray:
    """Rotate every frequency pair (x_i, x_{i+D/2}) by angle_i (broadcast over leading dims).

    Pair layout: frequency i pairs element i with element i + D/2 (the
    half-split layout of Qwen2.5-VL), rotated counter-clockwise:
        (x_i, x_{i+D/2}) -> (x_i cos a - x_{i+D/2} sin a,  x_{i+D/2} cos a + x_i sin a).
    """
    h = x.shape[-1] // 2
    c, s = np.cos(angle), np.sin(angle)
    a, b = x[..., :h], x[..., h:]
    return np.concatenate([a * c - b * s, b * c + a * s], axis=-1)


def mrope_rotate(x, pos, base=1e6, sections=(16, 24, 24)) -> np.ndarray:
    """Eq. 2: f(x, p) = R(alpha(p)) x with alpha_i(p) = p_sigma(i) * theta_i.

    x: [..., D] (any float, computed in fp64); pos: [..., 3] integer (t, h, w),
    broadcast against x's leading dimensions.
    """
    x = np.asarray(x, dtype=np.float64)
    pos = np.asarray(pos, dtype=np.float64)
    theta = rope_theta(base, x.shape[-1])
    sig = axis_of_pair(sections)
    angle = pos[..., sig] * theta                       # [..., D/2]
    return _rotate_pairs(x, angle)


# ----------------------------------------------------------------------------
# Eq. 3: delta re-base of stored post-rotary keys
# ----------------------------------------------------------------------------


def rebase_f64(k, pos_from, pos_to, base=1e6, sections=(16, 24, 24)) -> np.ndarray:
    """Eq. 3: R(Delta) f(x, p) with Delta_i = (p'_sigma(i) - p_sigma(i)) * theta_i, in fp64.

    k: [..., T, H, D] stored keys; pos_from, pos_to: [T, 3] integer
    coordinates.  Values are never rotated (Sec. 2).  Works for any leading
    dims (layers) and any head count: the angle depends only on the token.
    """
    k = np.asarray(k, dtype=np.float64)
    d = np.asarray(pos_to, dtype=np.int64) - np.asarray(pos_from, dtype=np.int64)   # [T, 3]
    theta = rope_theta(base, k.shape[-1])
    sig = axis_of_pair(sections)
    angle = d[:, sig].astype(np.float64) * theta        # [T, D/2]
    return _rotate_pairs(k, angle[:, None, :])          # broadcast over heads and layers


def round_to_bf16(x) -> np.ndarray:
    """Round to the nearest bfloat16 value, ties to even; returns the value as fp64.

    bfloat16 keeps 8 significant bits and fp32's exponent range, so the
    rounding quantum of a value in [2^(e-1), 2^e) is 2^(e-8), and never below
    2^-133 (its subnormal spacing).  Values too large round to +-inf.
    """
    x = np.asarray(x, dtype=np.float64)
    _, e = np.frexp(x)
    qexp = np.maximum(e - 8, -133)
    with np.errstate(over="ignore", invalid="ignore"):
        r = np.rint(np.ldexp(x, -qexp))                 # round half to even
        y = np.ldexp(r, qexp)
    big = np.abs(y) >= 2.0 ** 128
    return np.where(np.isfinite(x) & big, np.copysign(np.inf, x), y)


def bf16_bits(x) -> np.ndarray:
    """uint16 bit patterns of values that are exact bfloat16 numbers."""
    f = np.asarray(x, dtype=np.float64).astype(np.float32)
    return (f.view(np.uint32) >> 16).astype(np.uint16)


def bf16_from_bits(b) -> np.ndarray:
    """fp64 values of uint16 bfloat16 bit patterns."""
    u = np.asarray(b, dtype=np.uint16).astype(np.uint32) << 16
    return u.view(np.float32).astype(np.float64)


def round_to_storage(x, dtype: str) -> np.ndarray:
    """Round an fp64 result to the storage dtype ("bf16" or "f32"), returned as fp64."""
    if dtype == "bf16":
        return round_to_bf16(x)
    if dtype == "f32":
        return np.asarray(x, dtype=np.float64).astype(np.float32).astype(np.float64)
    raise ValueError(dtype)


def rebase(k_stored, pos_from, pos_to, dtype: str, base=1e6, sections=(16, 24, 24)):
    """Eq. 3 applied to a stored cache: returns (rounded result, fp64 result).

    The rounded result is the exact rotation rounded once to the storage
    dtype.  Rows whose token has Delta = 0 are returned unchanged bit for bit
    (cos 0 = 1, sin 0 = 0 exactly).
    """
    exact = rebase_f64(k_stored, pos_from, pos_to, base, sections)
    return round_to_storage(exact, dtype), exact


def scalar1d_targets(T: int) -> np.ndarray:
    """Scalar re-index baseline (Sec. 2, Table 1): token i gets (i, i, i).

    Flattening the composed sequence into consecutive scalar positions gives
    every token its sequence slot on all three axes, so two patches of one
    frame get different "time" coordinates.
    """
    i = np.arange(T, dtype=np.int64)
    return np.stack([i, i, i], axis=1).astype(np.int32)


# ----------------------------------------------------------------------------
# Eq. 5: key-deviation score
# ----------------------------------------------------------------------------


def score_f64(k_fresh, k_cached) -> np.ndarray:
    """Eq. 5 squared: delta_t^2 = sum over all kv heads and dims of (k_fresh - k_stored)^2, fp64.

    Inputs [n, ...]; every element of a token's layer-1 key enters the norm.
    """
    a = np.asarray(k_fresh, dtype=np.float64).reshape(len(k_fresh), -1)
    b = np.asarray(k_cached, dtype=np.float64).reshape(len(k_cached), -1)
    return np.sum((a - b) ** 2, axis=1)


def score_f32_canonical(k_fresh, k_cached) -> np.ndarray:
    """Eq. 5 squared in fp32, summed in one fixed order; this is the value that is ranked.

    Each token's E = Hkv*D elements (the stored values, exact in fp32):
      d_j = fp32(a_j - b_j);  q_j = fp32(d_j * d_j)            (no fused multiply-add)
      blocks of 8 consecutive elements: ((q0+q1)+(q2+q3))+((q4+q5)+(q6+q7))
      block sums s[0..B) padded with +0 to a power of two P, then
      for m = P/2, P/4, ..., 1:  s[b] = s[b] + s[b+m]  for b < m;   result s[0].
    Every operation is one fp32 rounding, so the result is reproducible bit for bit.
    """
    a = np.asarray(k_fresh, dtype=np.float32).reshape(len(k_fresh), -1)
    b = np.asarray(k_cached, dtype=np.float32).reshape(len(k_cached), -1)
    n, E = a.shape
    if E % 8:
        raise ValueError("row length must be a multiple of 8")
    d = a - b
    q = d * d
    qb = q.reshape(n, E // 8, 8)
    s = (((qb[..., 0] + qb[..., 1]) + (qb[..., 2] + qb[..., 3]))
         + ((qb[..., 4] + qb[..., 5]) + (qb[..., 6] + qb[..., 7])))
    B = E // 8
    P = 1
    while P < B:
        P *= 2
    if P > B:
        s = np.concatenate([s, np.zeros((n, P - B), dtype=np.float32)], axis=1)
    m = P // 2
    while m >= 1:
        s = s[:, :m] + s[:, m:2 * m]
        m //= 2
    return s[:, 0].astype(np.float32)


# ----------------------------------------------------------------------------
# Sec. 2: top-rho selection
# ----------------------------------------------------------------------------


def k_from_rho(rho_bp: int, n_cand: int) -> int:
    """k = ceil(rho * N_c), rho in basis points, exact integer arithmetic."""
    return (int(rho_bp) * int(n_cand) + 9999) // 10000


def order_key(score_f32) -> np.ndarray:
    """Total order of fp32 scores as uint32: larger key = ranks higher.

    For non-negative scores (all deviations) this is the order of the raw bit
    patterns, i.e. of the values, with +inf above every finite value and a
    positive NaN above +inf.  Negative values order below -0 < +0.
    """
    u = np.asarray(score_f32, dtype=np.float32).view(np.uint32).astype(np.uint64)
    neg = (u & 0x80000000) != 0
    return np.where(neg, (~u) & 0xFFFFFFFF, u | 0x80000000).astype(np.uint32)


def select_topk(score_f32, k: int, idx_base: int = 0) -> np.ndarray:
    """The k candidates with the largest score, ties broken by the lower index.

    Sorts all candidates by (order_key descending, local index ascending),
    keeps the first k, adds idx_base (the global index of candidate 0) and
    returns them in ascending order (int32).
    """
    key = order_key(score_f32).astype(np.int64)
    n = key.shape[0]
    if not 0 <= k <= n:
        raise ValueError("k out of range")
    order = np.lexsort((np.arange(n), -key))      # primary: -key, secondary: index
    return (np.sort(order[:k]) + idx_base).astype(np.int32)


# ----------------------------------------------------------------------------
# Eq. 1 + Sec. 2: repair attention of the selected rows
# ----------------------------------------------------------------------------


def scatter_rows(cache, rows, idx) -> np.ndarray:
    """Scatter-back (Sec. 2): the recomputed tokens' fresh keys/values replace their stored rows.

    cache [L, T, ...], rows [L, n, ...], idx [n] distinct token indices in [0, T).
    Returns a new array with cache[l, idx[r]] = rows[l, r] for every layer and row.
    """
    out = np.array(cache, copy=True)
    idx = np.asarray(idx, dtype=np.int64)
    for r, t in enumerate(idx):
        out[:, t] = rows[:, r]
    return out


def repair_attention(q, k, v, qpos, scale=None, rows=None, layers=None):
    """Causal GQA attention of selected query rows over the composed cache, fp64.

    q: [L, M, Hq, D]; k, v: [L, T, Hkv, D]; qpos: [M] global sequence index of
    each query row.  Row r at layer l, head h attends to keys j <= qpos[r] of
    kv head h // (Hq/Hkv) (causal in global sequence order, itself included):
        O = softmax(q k^T * scale) V,   scale = 1/sqrt(D)  (Eq. 1).
    Two passes: the row maximum, then exponentials, their sum and the
    weighted sum of values.  `rows` / `layers` restrict the output to a sample;
    returns (O [len(layers), len(rows), Hq, D], LSE [len(layers), len(rows), Hq])
    with LSE the natural-log normaliser including the scale.
    """
    L, M, Hq, D = q.shape
    Hkv = k.shape[2]
    G = Hq // Hkv
    if scale is None:
        scale = 1.0 / np.sqrt(D)
    rows = np.arange(M) if rows is None else np.asarray(rows)
    layers = np.arange(L) if layers is None else np.asarray(layers)
    out = np.zeros((len(layers), len(rows), Hq, D), dtype=np.float64)
    lse = np.zeros((len(layers), len(rows), Hq), dtype=np.float64)
    for li, l in enumerate(layers):
        for ri, r in enumerate(rows):
            n = int(qpos[r]) + 1
            for g in range(Hkv):
                kk = np.asarray(k[l, :n, g, :], dtype=np.float64)     # [n, D]
                vv = np.asarray(v[l, :n, g, :], dtype=np.float64)
                qq = np.asarray(q[l, r, g * G:(g + 1) * G, :], dtype=np.float64)   # [G, D]
                s = (qq @ kk.T) * scale                               # [G, n]
                mx = s.max(axis=1, keepdims=True)
                p = np.exp(s - mx)
                den = p.sum(axis=1, keepdims=True)
                out[li, ri, g * G:(g + 1) * G, :] = (p @ vv) / den
                lse[li, ri, g * G:(g + 1) * G] = (mx + np.log(den))[:, 0]
    return out, lse


__all__ = ["rope_theta", "axis_of_pair", "mrope_rotate", "rebase_f64", "rebase",
           "round_to_bf16", "round_to_storage", "bf16_bits", "bf16_from_bits",
           "scalar1d_targets", "score_f64", "score_f32_canonical", "k_from_rho",
           "order_key", "select_topk", "repair_attention"]
