"""AVTP pruning-stage oracle: a plain, slow, fp64 CPU restatement of the method.

TEST INFRASTRUCTURE. Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``
(its ``cpu_baseline`` leg and its ``--impl reference`` arm) may import or run this
module. The product path (``paper_2608_26806_gb300`` and its CUDA library) never
does, and this module imports nothing from it: the two share no code.

What it computes (paper: "Multi-Image Visual Token Pruning in Large Visual
Language Models", AVTP):

1A. Token importance from hidden-state variation (§3.3.1):
    ``I_v = 1 - Sim(h^l_v, h^prior_v)``; ``Sim`` is read as cosine similarity with
    each norm guarded below by 1e-8.
1B. Text-to-visual attention importance (the attention quantity of §3.3.2, kept
    per visual token): for each visual key t of request r,
    ``s_t = 1/(Hq*|Q_r|) * sum_h sum_{q in Q_r, q >= t} softmax_{h,q}(t)``, where
    Q_r are the request's text tokens, the softmax runs over the keys causally
    visible to q inside the request, logits are ``scale * q_h . k_{g(h)}`` and
    ``g(h) = h // (Hq/Hkv)`` (grouped-query attention).
2.  Per-image mean importance and adaptive keep ratio (§3.3.3):
    ``Ibar_i = mean_{v in V_i} I_v``, ``r_i = r_base + alpha*(Ibar_i - Ibar_avg)``,
    clamped to [5%, 95%] (App. A.2), then integer budgets whose total is the
    request's global budget.
3.  Per image, keep the ``k_i`` most important visual tokens; text is kept (§3.1,
    §3.3.3); the result is an order-preserving subsequence (§3.1).
4.  Compaction: a row gather of the kept tokens (§3.1, ``E_pruned = p(E_v)``).
5.  The layout of the pruned batch, on which the stage runs again at a later layer in
    a progressive schedule (§3.3.2), with the compacted hidden states of this pruning
    point as that layer's h_prior (§3.3.1).
6.  Pruning-layer selection (§3.3.2): per sample and layer the attention mass on the
    visual tokens, the per-sample ranking of the layers, the mean rank, the top-k layers.
    The attention of step 1B may also take the request's last token as its only query
    (§4.1, the output token's attention that FAST-V ranks by).
7.  The pruning layer's attention forward (the FlashAttention-style pass whose
    normaliser and probabilities criterion 1B reuses, §3.2): for every token of a
    request and every head, ``O = softmax(scale * q K^T) V`` over the causally visible
    keys of the request, and its natural-log normaliser.

Readings of points the paper leaves open (each is also listed with its reason in
the design notes of the repository):

* Per-image sums are taken in fixed point, ``S_i = sum rint(fx(I_t) * 2^32)`` on the
  fp32-rounded score, with ``fx`` mapping NaN to 0 and clamping to +-2^10, so that
  every summation order gives the same integer.
* ``Ibar_avg`` is the token-weighted mean ``sum_i S_i / 2^32 / N_vis``.
* The budget rule is computed in exact rational arithmetic (``fractions.Fraction``):
  the means, the ratios, the shift and the kept masses are the plain formulas, and the
  fp32 parameters (keep ratio, alpha, clamps) enter as the exact values they hold.
* The global budget is ``B_r = floor(keep_ratio_r * N_vis_r + 1/2)``.
* ``relative=1`` replaces the additive rule by ``r_i = r_base*(1 + alpha*(Ibar_i/Ibar_avg - 1))``
  (``r_base`` when ``Ibar_avg == 0``); criterion 1B's raw values are of order
  1/N, where the additive rule would leave every ratio at ``r_base``.
* A shift lambda (water-fill) restores the clamped total:
  ``sum_i n_i * clamp(r_i + lambda, r_min, r_max) = B_r``; when B_r lies outside
  ``[N r_min, N r_max]`` every image takes the nearer clamp.
* Integer budgets: ``x_i = n_i * clamp(r_i + lambda)``, ``k_i = min(floor(x_i), n_i)``,
  then largest remainder (ties to the lower image index) until ``sum k_i = B_r``; a
  surplus is removed from the smallest remainders (ties to the higher index).
* Top-k order: score descending, position ascending; NaN ranks below -inf;
  -0 equals +0.
"""
from __future__ import annotations

import math
from fractions import Fraction
from typing import Dict, List, Optional, Sequence

import numpy as np

FX_FRAC_BITS = 32
FX_SCORE_LIMIT = 1024.0  # |score| is clamped to 2^10 before the fixed-point conversion
NORM_EPS = 1e-8
SUM_MAGNITUDE_BITS = 42  # |S_i| <= n_i * 2^42: scores clamped to +-2^10, 32 fraction bits


# ----------------------------------------------------------------------------
# helpers
# ----------------------------------------------------------------------------
def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    """Decode bf16 bit patterns (uint16) to fp64 (exact widening).

    Input decoding only, not a step of the paper's method.
    """
    u = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return u.view(np.float32).astype(np.float64)


def _image_rows(layout, r: int, i: int) -> np.ndarray:
    base = int(layout.cu_seqlens[r]) + int(layout.img_start[i])
    return np.arange(base, base + int(layout.img_len[i]), dtype=np.int64)


def _request_visual_local(layout, r: int) -> np.ndarray:
    """Boolean mask over the request's local positions: True inside an image span."""
    T_r = int(layout.cu_seqlens[r + 1]) - int(layout.cu_seqlens[r])
    m = np.zeros(T_r, dtype=bool)
    for i in range(int(layout.img_cu[r]), int(layout.img_cu[r + 1])):
        s = int(layout.img_start[i])
        m[s:s + int(layout.img_len[i])] = True
    return m


# ----------------------------------------------------------------------------
# Step 1A: hidden-state variation (paper §3.3.1)
# ----------------------------------------------------------------------------
def score_hidden_variation(layout, h_cur: np.ndarray, h_prior: np.ndarray) -> np.ndarray:
    """``I_v = 1 - cos(h^l_v, h^prior_v)`` for every visual token (fp64); text entries are 0.

    ``h_cur`` / ``h_prior``: bf16 bits [T, D]. Paper §3.3.1 (importance score).
    """
    T = int(layout.cu_seqlens[-1])
    out = np.zeros(T, dtype=np.float64)
    for r in range(len(layout.cu_seqlens) - 1):
        for i in range(int(layout.img_cu[r]), int(layout.img_cu[r + 1])):
            rows = _image_rows(layout, r, i)
            a = bf16_to_f64(h_cur[rows])
            b = bf16_to_f64(h_prior[rows])
            dot = np.sum(a * b, axis=1)
            na = np.sqrt(np.sum(a * a, axis=1))
            nb = np.sqrt(np.sum(b * b, axis=1))
            cos = dot / (np.maximum(na, NORM_EPS) * np.maximum(nb, NORM_EPS))
            out[rows] = 1.0 - cos
    return out


# ----------------------------------------------------------------------------
# Step 1B: text-to-visual attention (attention quantity of paper §3.3.2)
# ----------------------------------------------------------------------------
QUERY_SETS = ("text", "last", "all")


def query_positions(layout, r: int, query_set: str = "text") -> np.ndarray:
    """Request-local positions of the queries whose attention scores the visual keys.

    ``"text"``: every text token of the request (the attention of §3.3.2 kept per token).
    ``"last"``: the request's last token alone, the token whose output predicts the first
    generated token (the attention FAST-V ranks visual tokens by, §4.1).
    ``"all"``: every token of the request (the attention forward of the layer, §3.2).
    """
    T_r = int(layout.cu_seqlens[r + 1]) - int(layout.cu_seqlens[r])
    if query_set == "text":
        return np.nonzero(~_request_visual_local(layout, r))[0]
    if query_set == "last":
        return np.arange(T_r - 1, T_r) if T_r > 0 else np.zeros(0, dtype=np.int64)
    if query_set == "all":
        return np.arange(T_r)
    raise ValueError(query_set)


def attention_logits(layout, q, k, r: int, h: int, n_q_heads: int, n_kv_heads: int, scale: float,
                     query_set: str = "text"):
    """Scaled logits of request r, head h: the query set's rows x all request keys.
    Follows paper §3.3.2, the attention of text queries to visual tokens; grouped-query heads.

    Returns ``(z, qpos)``; ``z`` is fp64 [|Q_r|, T_r] with ``-inf`` where the key
    lies after the query (causal mask); ``qpos`` the queries' request-local positions.
    """
    a = int(layout.cu_seqlens[r])
    b = int(layout.cu_seqlens[r + 1])
    qpos = query_positions(layout, r, query_set)
    g = h // (n_q_heads // n_kv_heads)
    Qh = bf16_to_f64(q[a + qpos, h, :])              # [nq, d]
    Kg = bf16_to_f64(k[a:b, g, :])                   # [T_r, d]
    z = float(scale) * (Qh @ Kg.T)                   # [nq, T_r]
    keys = np.arange(b - a)
    visible = keys[None, :] <= qpos[:, None]
    z = np.where(visible, z, -np.inf)
    return z, qpos


def logsumexp_rows(z: np.ndarray) -> np.ndarray:
    """Natural-log sum of exp over each row, with max subtraction.

    Follows paper §3.3.2, the softmax normaliser.
    """
    m = np.max(z, axis=1)
    return m + np.log(np.sum(np.exp(z - m[:, None]), axis=1))


def text_lse(layout, q, k, n_q_heads: int, n_kv_heads: int, scale: float, query_set: str = "text") -> np.ndarray:
    """Per (head, query) natural-log LSE of the scaled causal logits: fp64 [Hq, T].
    Follows paper §3.3.2; the normaliser a FlashAttention forward also returns (§3.2).

    This is the normaliser a FlashAttention-style forward pass keeps per query row;
    the entries of tokens outside the query set are left 0.
    """
    T = int(layout.cu_seqlens[-1])
    out = np.zeros((n_q_heads, T), dtype=np.float64)
    for r in range(len(layout.cu_seqlens) - 1):
        a = int(layout.cu_seqlens[r])
        for h in range(n_q_heads):
            z, qpos = attention_logits(layout, q, k, r, h, n_q_heads, n_kv_heads, scale, query_set)
            if qpos.size:
                out[h, a + qpos] = logsumexp_rows(z)
    return out


def score_text_attention(layout, q, k, n_q_heads: int, n_kv_heads: int, scale: float,
                         lse: Optional[np.ndarray] = None, query_set: str = "text") -> np.ndarray:
    """Mean over heads and queries of the causal softmax probability of each visual key.
    Follows paper §3.3.2, the attention quantity kept per visual token; with
    ``query_set="last"``, §4.1's attention of the output token.

    ``q``: bf16 bits [T, Hq, d]; ``k``: bf16 bits [T, Hkv, d]; ``lse`` (optional) [Hq, T]
    natural-log normalisers for the query rows; when given they replace the
    oracle's own. Returns fp64 [T] (non-visual entries 0).
    """
    T = int(layout.cu_seqlens[-1])
    out = np.zeros(T, dtype=np.float64)
    for r in range(len(layout.cu_seqlens) - 1):
        a = int(layout.cu_seqlens[r])
        b = int(layout.cu_seqlens[r + 1])
        vis = _request_visual_local(layout, r)
        nq = len(query_positions(layout, r, query_set))
        if nq == 0:
            continue
        acc = np.zeros(b - a, dtype=np.float64)
        for h in range(n_q_heads):
            z, qpos = attention_logits(layout, q, k, r, h, n_q_heads, n_kv_heads, scale, query_set)
            if lse is None:
                norm = logsumexp_rows(z)
            else:
                norm = np.asarray(lse, dtype=np.float64)[h, a + qpos]
            P = np.exp(z - norm[:, None])  # exp(-inf) = 0 on masked keys
            acc += np.sum(P, axis=0)
        out[a:b][vis] = acc[vis] / (n_q_heads * nq)
    return out


# ----------------------------------------------------------------------------
# Step 2: per-image sums, adaptive ratios and integer budgets (paper §3.3.3, App. A.2)
# ----------------------------------------------------------------------------
def to_fp32(scores: np.ndarray) -> np.ndarray:
    """The interface type of scores is fp32 (round to nearest).

    The paper fixes no precision; fp32 is the scores' type at the library boundary.
    """
    return np.asarray(scores, dtype=np.float64).astype(np.float32)


def fixed_point(scores_f32: np.ndarray) -> np.ndarray:
    """``rint(fx(s) * 2^32)`` as int64; fx: NaN -> 0, clamp to [-2^10, 2^10].

    Follows paper §3.3.3, the terms of the per-image sums.
    """
    s = np.asarray(scores_f32, dtype=np.float32).astype(np.float64)
    s = np.where(np.isnan(s), 0.0, s)
    s = np.clip(s, -FX_SCORE_LIMIT, FX_SCORE_LIMIT)
    return np.rint(s * float(2 ** FX_FRAC_BITS)).astype(np.int64)



def attention_forward(layout, q, k, v, n_q_heads: int, n_kv_heads: int, scale: float):
    """The layer's causal attention forward: ``O = softmax(scale * q K^T) V`` per token and
    head over the request's causally visible keys, with the natural-log normaliser.
    Follows paper §3.2 (the FlashAttention-style forward whose normaliser criterion 1B
    reuses) and §3.3.2 (grouped-query heads ``g(h) = h // (Hq/Hkv)``).

    ``q``: bf16 bits [T, Hq, d]; ``k``, ``v``: bf16 bits [T, Hkv, d]. Returns ``(O, lse)``:
    fp64 [T, Hq, d] and fp64 [Hq, T].
    """
    T = int(layout.cu_seqlens[-1])
    d = q.shape[2]
    O = np.zeros((T, n_q_heads, d), dtype=np.float64)
    lse = np.zeros((n_q_heads, T), dtype=np.float64)
    G = n_q_heads // n_kv_heads
    for r in range(len(layout.cu_seqlens) - 1):
        a = int(layout.cu_seqlens[r])
        b = int(layout.cu_seqlens[r + 1])
        if b == a:
            continue
        for h in range(n_q_heads):
            z, qpos = attention_logits(layout, q, k, r, h, n_q_heads, n_kv_heads, scale, "all")
            norm = logsumexp_rows(z)
            P = np.exp(z - norm[:, None])                       # [T_r, T_r], rows sum to 1
            O[a + qpos, h, :] = P @ bf16_to_f64(v[a:b, h // G, :])
            lse[h, a + qpos] = norm
    return O, lse


def attention_forward_rows(layout, q, k, v, n_q_heads: int, n_kv_heads: int, scale: float, r: int,
                           rows: Sequence[int]):
    """The attention forward of `attention_forward` for a few request-local query rows of
    request r only (for workloads too large to run whole). Returns ``(O, lse)``:
    fp64 [len(rows), Hq, d] and fp64 [Hq, len(rows)].
    """
    a = int(layout.cu_seqlens[r])
    rows = np.asarray(rows, dtype=np.int64)
    d = q.shape[2]
    G = n_q_heads // n_kv_heads
    O = np.zeros((len(rows), n_q_heads, d), dtype=np.float64)
    lse = np.zeros((n_q_heads, len(rows)), dtype=np.float64)
    for j, p in enumerate(rows):
        for h in range(n_q_heads):
            g = h // G
            qv = bf16_to_f64(q[a + p, h, :])
            Kg = bf16_to_f64(k[a:a + p + 1, g, :])                # keys 0..p of the request
            z = float(scale) * (Kg @ qv)
            m = np.max(z)
            w = np.exp(z - m)
            O[j, h, :] = (w / np.sum(w)) @ bf16_to_f64(v[a:a + p + 1, g, :])
            lse[h, j] = m + np.log(np.sum(w))
    return O, lse

def image_sums(layout, scores_f32: np.ndarray) -> np.ndarray:
    """Fixed-point per-image sums ``S_i`` (int64 [n_img]) of the fp32 scores.

    Follows paper §3.3.3, the sums behind the mean importance Ibar_i.
    """
    fx = fixed_point(scores_f32)
    n_img = len(layout.img_len)
    out = np.zeros(n_img, dtype=np.int64)
    for r in range(len(layout.cu_seqlens) - 1):
        for i in range(int(layout.img_cu[r]), int(layout.img_cu[r + 1])):
            out[i] = int(sum(int(v) for v in fx[_image_rows(layout, r, i)]))
    return out


def global_budget(keep_ratio_f32: float, n_vis: int) -> int:
    """``B_r = floor(keep_ratio * N_vis + 1/2)``, the fp32 ratio taken exactly.

    Follows paper §3.3.3 and §4.1, the request's keep ratio.
    """
    return math.floor(Fraction(float(np.float32(keep_ratio_f32))) * int(n_vis) + Fraction(1, 2))


def _clamp(x, lo, hi):
    return min(max(x, lo), hi)


def image_means(S: Sequence[int], n: Sequence[int]) -> List[Fraction]:
    """``Ibar_i = S_i / (2^32 n_i)``: the mean importance of each image, exactly.

    Follows paper §3.3.3, the mean importance of an image.
    """
    return [Fraction(int(S[i]), (1 << FX_FRAC_BITS) * int(n[i])) for i in range(len(n))]


def average_importance(S: Sequence[int], n: Sequence[int]) -> Fraction:
    """``Ibar_avg = sum_i S_i / (2^32 N_vis)``, the token-weighted mean over the request's images.

    Follows paper §3.3.3, the average importance across images (token-weighted reading).
    """
    return Fraction(sum(int(v) for v in S), (1 << FX_FRAC_BITS) * sum(int(v) for v in n))


def adaptive_ratios(S: Sequence[int], n: Sequence[int], r_base_f32, alpha_f32, relative: bool) -> List[Fraction]:
    """The adaptive keep ratio of every image, before the clamps, as exact rationals.

    Follows paper §3.3.3: ``r_i = r_base + alpha * (Ibar_i - Ibar_avg)``; with ``relative``,
    ``r_i = r_base * (1 + alpha * (Ibar_i / Ibar_avg - 1))`` (``r_base`` when ``Ibar_avg == 0``).
    The fp32 parameters enter as the exact values they hold.
    """
    r_base = Fraction(float(np.float32(r_base_f32)))
    alpha = Fraction(float(np.float32(alpha_f32)))
    ibar = image_means(S, n)
    avg = average_importance(S, n)
    if not relative:
        return [r_base + alpha * (ib - avg) for ib in ibar]
    if avg == 0:
        return [r_base for _ in ibar]
    return [r_base * (1 + alpha * (ib / avg - 1)) for ib in ibar]


def clamped_total(r: Sequence[Fraction], n: Sequence[int], lam: Fraction, r_min: Fraction, r_max: Fraction) -> Fraction:
    """``G(lambda) = sum_i n_i * clamp(r_i + lambda, r_min, r_max)``: the kept total after a shift.

    Follows paper App. A.2, the ratios clamped to [r_min, r_max].
    """
    return sum((int(n[i]) * _clamp(r[i] + lam, r_min, r_max) for i in range(len(n))), Fraction(0))


def water_fill(r: Sequence[Fraction], n: Sequence[int], B: int, r_min: Fraction, r_max: Fraction) -> Fraction:
    """The shift lambda that restores the request's budget after the clamps: ``G(lambda) = B``.
    Follows paper App. A.2, clamped ratios with the global total kept.

    G is continuous, non-decreasing and linear between the breakpoints ``r_min - r_i`` and
    ``r_max - r_i``. Below the lowest breakpoint every image sits at ``r_min`` and above the
    highest at ``r_max``; when B lies outside ``[N r_min, N r_max]`` the nearer end is
    returned (every image at that clamp). Otherwise lambda is the point where the linear
    piece between the two breakpoints that bracket B reaches B; where G is flat at B
    (every image clamped) any such point gives the same clamped ratios.
    """
    pts = sorted(set([r_min - v for v in r] + [r_max - v for v in r]))
    G = [clamped_total(r, n, p, r_min, r_max) for p in pts]
    if B <= G[0]:
        return pts[0]
    if B >= G[-1]:
        return pts[-1]
    for k in range(len(pts) - 1):
        if G[k] < B <= G[k + 1]:
            return pts[k] + (B - G[k]) * (pts[k + 1] - pts[k]) / (G[k + 1] - G[k])
    raise AssertionError("unreachable: G is non-decreasing and B lies within its range")


def integer_budgets(x: Sequence[Fraction], n: Sequence[int], B: int) -> List[int]:
    """Largest-remainder rounding of the kept masses ``x_i`` to integers summing to B.
    Follows paper §3.3.3, integer budgets whose total is the global budget.

    ``k_i = floor(x_i)``; while the total is short, one more token goes to each of the
    images still below ``n_i`` with the largest ``x_i - floor(x_i)`` (ties to the lower
    index); while it is over, one token is taken from the images above 0 with the
    smallest remainders (ties to the higher index).
    """
    m = len(n)
    k = [min(math.floor(v), int(n[i])) for i, v in enumerate(x)]
    frac = [v - math.floor(v) for v in x]
    while sum(k) < B:
        need = B - sum(k)
        elig = [i for i in range(m) if k[i] < int(n[i])]
        order = sorted(elig, key=lambda i: (-frac[i], i))
        for i in order[:need]:
            k[i] += 1
    while sum(k) > B:
        extra = sum(k) - B
        elig = [i for i in range(m) if k[i] > 0]
        order = sorted(elig, key=lambda i: (frac[i], -i))
        for i in order[:extra]:
            k[i] -= 1
    return k


def allocate(layout, S: np.ndarray, keep_ratio: np.ndarray, alpha: float = 1.0,
             r_min: float = 0.05, r_max: float = 0.95, relative: bool = False) -> Dict[str, np.ndarray]:
    """Per-image budgets ``k_i`` and the packed output offsets ``out_cu_seqlens``.
    Follows paper §3.3.3 with the clamps of App. A.2, in exact rational arithmetic.

    Per request: ``B = floor(r_base N_vis + 1/2)``; the ratios of ``adaptive_ratios``;
    the shift of ``water_fill``; ``x_i = n_i clamp(r_i + lambda, r_min, r_max)``; the
    integers of ``integer_budgets``. The sums must satisfy ``|S_i| <= n_i * 2^42`` (every
    fixed-point score is within +-2^42), and every keep ratio must lie within the clamps
    ``[r_min, r_max]`` (else no ratio shift meets both the clamps and the global budget);
    otherwise ValueError. Returns ``budgets`` int32 [n_img], ``out_cu_seqlens`` int32 [R+1]
    and, for inspection, ``ratios`` (before the clamps) and ``lam`` per request, as floats.
    """
    R = len(layout.cu_seqlens) - 1
    fr_min = Fraction(float(np.float32(r_min)))
    fr_max = Fraction(float(np.float32(r_max)))
    budgets = np.zeros(len(layout.img_len), dtype=np.int32)
    out_cu = np.zeros(R + 1, dtype=np.int32)
    ratios = np.zeros(len(layout.img_len), dtype=np.float64)
    lams = np.zeros(R, dtype=np.float64)
    for rq in range(R):
        i0, i1 = int(layout.img_cu[rq]), int(layout.img_cu[rq + 1])
        n = [int(v) for v in layout.img_len[i0:i1]]
        n_vis = sum(n)
        T_r = int(layout.cu_seqlens[rq + 1]) - int(layout.cu_seqlens[rq])
        n_txt = T_r - n_vis
        r_base = Fraction(float(np.float32(keep_ratio[rq])))
        if not (fr_min <= r_base <= fr_max):
            raise ValueError(f"request {rq}: keep ratio {float(r_base)} outside the clamps [{r_min}, {r_max}]")
        B = global_budget(keep_ratio[rq], n_vis)
        if i1 > i0:
            Sr = [int(v) for v in S[i0:i1]]
            for j in range(len(n)):
                if abs(Sr[j]) > n[j] << SUM_MAGNITUDE_BITS:
                    raise ValueError(f"image {i0 + j}: |S_i| exceeds n_i * 2^{SUM_MAGNITUDE_BITS}")
            r = adaptive_ratios(Sr, n, keep_ratio[rq], alpha, relative)
            lam = water_fill(r, n, B, fr_min, fr_max)
            x = [n[i] * _clamp(r[i] + lam, fr_min, fr_max) for i in range(len(n))]
            budgets[i0:i1] = integer_budgets(x, n, B)
            ratios[i0:i1] = [float(v) for v in r]
            lams[rq] = float(lam)
        out_cu[rq + 1] = out_cu[rq] + B + n_txt
    return {"budgets": budgets, "out_cu_seqlens": out_cu, "ratios": ratios, "lam": lams}


# ----------------------------------------------------------------------------
# Step 3: per-image top-k, text kept, ascending order (paper §3.1, §3.3.3)
# ----------------------------------------------------------------------------
def rank_key(score: float, pos: int):
    """Sort key: score descending, position ascending; NaN below every number.

    Follows paper §3.3.3, the most important tokens first.
    """
    if math.isnan(score):
        return (1, 0.0, pos)
    return (0, -score, pos)


def select(layout, scores_f32: np.ndarray, budgets: np.ndarray) -> np.ndarray:
    """Packed global indices of the kept tokens (int32), ascending within each request.

    Follows paper §3.1, an order-preserving subsequence; §3.3.3, k_i tokens per image.
    """
    sc = np.asarray(scores_f32, dtype=np.float32)
    kept: List[int] = []
    for r in range(len(layout.cu_seqlens) - 1):
        a = int(layout.cu_seqlens[r])
        b = int(layout.cu_seqlens[r + 1])
        keep = ~_request_visual_local(layout, r)  # text always kept
        for i in range(int(layout.img_cu[r]), int(layout.img_cu[r + 1])):
            rows = _image_rows(layout, r, i)
            order = sorted(rows.tolist(), key=lambda t: rank_key(float(sc[t]), t))
            for t in order[:int(budgets[i])]:
                keep[t - a] = True
        kept.extend((np.nonzero(keep)[0] + a).tolist())
    return np.asarray(kept, dtype=np.int32)


# ----------------------------------------------------------------------------
# Step 4: compaction (paper §3.1)
# ----------------------------------------------------------------------------
def compact(kept_idx: np.ndarray, rows: np.ndarray) -> np.ndarray:
    """``out[j] = rows[kept_idx[j]]`` along axis 0 (any dtype, bit-exact).

    Follows paper §3.1, E_pruned = p(E_v).
    """
    return np.asarray(rows)[np.asarray(kept_idx, dtype=np.int64)]


def compact_planes(kept_idx: np.ndarray, planes: np.ndarray) -> np.ndarray:
    """Gather along the token axis of a [P, T] array (e.g. M-RoPE position ids).

    Follows paper §3.1, the position ids of the kept tokens.
    """
    return np.asarray(planes)[:, np.asarray(kept_idx, dtype=np.int64)]


# ----------------------------------------------------------------------------
# Layout of the pruned batch (progressive pruning, paper §3.3.2: the stage runs again
# at later layers on the shortened sequence, with the previous pruning point's hidden
# states as h_prior, §3.3.1)
# ----------------------------------------------------------------------------
def pruned_layout(layout, kept_idx: np.ndarray, out_cu_seqlens: np.ndarray) -> Dict[str, np.ndarray]:
    """Image spans of the pruned batch, read off the kept tokens.
    Follows paper §3.3.2, the progressive schedule; §3.3.1, h_prior.

    In request r of the pruned batch, image i starts at the number of kept tokens of the
    request that lie before the image's span, and holds the kept tokens inside the span
    (its budget). Requests and their image lists are unchanged. Returns cu_seqlens,
    img_cu, img_start and img_len (int32) of the pruned batch.
    """
    kept = np.asarray(kept_idx, dtype=np.int64)
    cu2 = np.asarray(out_cu_seqlens, dtype=np.int64)
    starts, lens = [], []
    for r in range(len(layout.cu_seqlens) - 1):
        a = int(layout.cu_seqlens[r])
        local = kept[cu2[r]:cu2[r + 1]] - a  # request-local positions of the kept tokens
        for i in range(int(layout.img_cu[r]), int(layout.img_cu[r + 1])):
            s0 = int(layout.img_start[i])
            s1 = s0 + int(layout.img_len[i])
            starts.append(int(np.count_nonzero(local < s0)))
            lens.append(int(np.count_nonzero((local >= s0) & (local < s1))))
    return {"cu_seqlens": cu2.astype(np.int32), "img_cu": np.asarray(layout.img_cu, dtype=np.int32).copy(),
            "img_start": np.asarray(starts, dtype=np.int32), "img_len": np.asarray(lens, dtype=np.int32)}


# ----------------------------------------------------------------------------
# Pruning-layer selection (paper §3.3.2): the layers whose attention to visual tokens
# ranks highest across sample requests
# ----------------------------------------------------------------------------
def layer_attention(layout, img_sums: np.ndarray) -> np.ndarray:
    """``A_l^(i) = sum_j Attention(l, v_j)`` of one layer for every request (sample) i.
    Follows paper §3.3.2, the cumulative attention a layer assigns to the visual tokens.

    ``Attention(l, v_j)`` is read as the text-attention score of token ``v_j`` at layer l
    (``score_text_attention``), so ``A`` is the sum of the request's fixed-point per-image
    sums of that criterion: int64 [R], units of 2^-32.
    """
    R = len(layout.cu_seqlens) - 1
    out = np.zeros(R, dtype=np.int64)
    for r in range(R):
        out[r] = sum(int(v) for v in img_sums[int(layout.img_cu[r]):int(layout.img_cu[r + 1])])
    return out


def layer_ranks(A: np.ndarray) -> np.ndarray:
    """``Rank(A_l^(i))``: per sample, the rank of each of the L layers, 1 for the most attention.
    Follows paper §3.3.2, the per-sample ranking of the layers.

    ``A``: int [N, L]. Equal values rank by the lower layer index, so each sample's ranks
    are a permutation of 1..L. Returns int64 [N, L].
    """
    A = np.asarray(A)
    N, L = A.shape
    ranks = np.zeros((N, L), dtype=np.int64)
    for i in range(N):
        order = sorted(range(L), key=lambda l: (-int(A[i, l]), l))
        for p, l in enumerate(order):
            ranks[i, l] = p + 1
    return ranks


def mean_ranks(A: np.ndarray):
    """``R_l = (1/N) sum_i Rank(A_l^(i))``, with the exact integer sum of ranks beside it.
    Follows paper §3.3.2, the average ranking across the samples.

    Returns ``(rank_sum int64 [L], R fp64 [L])``.
    """
    ranks = layer_ranks(A)
    rank_sum = ranks.sum(axis=0).astype(np.int64)
    return rank_sum, rank_sum / float(ranks.shape[0])


def select_layers(A: np.ndarray, k: int) -> np.ndarray:
    """The k pruning layers: the best (lowest) average ranks, ties to the lower layer index.
    Follows paper §3.3.2, the top-k layers chosen as pruning layers.

    Returns int32 [k], best first.
    """
    rank_sum, _ = mean_ranks(A)
    order = sorted(range(len(rank_sum)), key=lambda l: (int(rank_sum[l]), l))
    return np.asarray(order[:k], dtype=np.int32)


# ----------------------------------------------------------------------------
# The whole stage
# ----------------------------------------------------------------------------
def prune(layout, *, criterion: str = "hidden_variation", keep_ratio, alpha: float = 1.0,
          r_min: float = 0.05, r_max: float = 0.95, relative: Optional[bool] = None,
          h_cur=None, h_prior=None, q=None, k=None, n_q_heads=None, n_kv_heads=None,
          scale=None, lse=None, scores_f32=None, rows: Optional[Dict[str, np.ndarray]] = None,
          planes: Optional[Dict[str, np.ndarray]] = None) -> Dict[str, np.ndarray]:
    """score -> per-image sums -> budgets -> selection -> compaction.
    Follows paper §3.1-§3.3, the whole stage.

    ``scores_f32`` (optional) replaces step 1, to run steps 2-4 on given scores.
    ``rows``: name -> [T, ...] arrays gathered along axis 0; ``planes``: name ->
    [P, T] arrays gathered along axis 1. ``relative`` defaults to False for the
    hidden-variation criterion and True for text attention.
    """
    if relative is None:
        relative = criterion != "hidden_variation"
    if scores_f32 is None:
        if criterion == "hidden_variation":
            s64 = score_hidden_variation(layout, h_cur, h_prior)
        elif criterion == "text_attention":
            s64 = score_text_attention(layout, q, k, n_q_heads, n_kv_heads, scale, lse=lse)
        else:
            raise ValueError(criterion)
        scores_f32 = to_fp32(s64)
    S = image_sums(layout, scores_f32)
    alloc = allocate(layout, S, keep_ratio, alpha, r_min, r_max, relative)
    kept = select(layout, scores_f32, alloc["budgets"])
    out = {"scores": scores_f32, "img_sums": S, "budgets": alloc["budgets"],
           "out_cu_seqlens": alloc["out_cu_seqlens"], "kept_idx": kept}
    for name, arr in (rows or {}).items():
        out[name] = compact(kept, arr)
    for name, arr in (planes or {}).items():
        out[name] = compact_planes(kept, arr)
    return out
