"""Pins of the fp64 oracle against what the paper and the mathematics fix.

Nothing here compares the oracle with itself: each check uses a hand-derived
value (tests/golden), a closed form, a library routine reached by a different
route (scipy cosine distance, scipy softmax over the full square attention
matrix with np.repeat for the grouped heads), brute-force enumeration, or an
invariant the method must satisfy. CPU only.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest
import scipy.spatial.distance as ssd
import scipy.special as ssp

from oracle import avtp_oracle as O
from paper_2608_26806_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _load(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def _f(v):
    return float(v) if not isinstance(v, str) else float(v.replace("inf", "inf"))


def _bits(rows):
    return synth.f32_to_bf16_bits(np.asarray(rows, dtype=np.float32))


# ---------------------------------------------------------------- step 1A
def test_hidden_variation_golden():
    g = _load("hidden_variation.json")
    for case in g["cases"]:
        lay = synth.Layout.from_segments([[("i", 1)]])
        I = O.score_hidden_variation(lay, _bits([case["h_cur"]]), _bits([case["h_prior"]]))
        assert I[0] == pytest.approx(case["expected"], abs=1e-15), case["derivation"]


def test_hidden_variation_matches_scipy_cosine_distance():
    rng = np.random.default_rng(0)
    lay = synth.Layout.from_segments([[("t", 3), ("i", 40), ("t", 2), ("i", 25)]])
    T, D = lay.n_tokens, 96
    hc = _bits(rng.standard_normal((T, D)))
    hp = _bits(rng.standard_normal((T, D)) * 0.3 + synth.bf16_bits_to_f32(hc))
    I = O.score_hidden_variation(lay, hc, hp)
    vis = lay.visual_mask()
    a = synth.bf16_bits_to_f32(hc).astype(np.float64)
    b = synth.bf16_bits_to_f32(hp).astype(np.float64)
    for t in range(T):
        if vis[t]:
            assert I[t] == pytest.approx(ssd.cosine(a[t], b[t]), rel=1e-12, abs=1e-14)
        else:
            assert I[t] == 0.0


def test_hidden_variation_identity_and_opposite():
    rng = np.random.default_rng(1)
    lay = synth.Layout.from_segments([[("i", 16)]])
    h = _bits(rng.standard_normal((16, 64)))
    assert np.allclose(O.score_hidden_variation(lay, h, h), 0.0, atol=1e-15)
    neg = (h ^ np.uint16(0x8000)).astype(np.uint16)  # bf16 negation flips the sign bit
    assert np.allclose(O.score_hidden_variation(lay, h, neg), 2.0, atol=1e-15)


# ---------------------------------------------------------------- step 1B
def test_text_attention_golden():
    g = _load("text_attention.json")
    lay = synth.Layout.from_segments([[(k, n) for k, n in g["layout"]]])
    q = _bits(g["q"]).reshape(-1, 1, 1)
    k = _bits(g["k"]).reshape(-1, 1, 1)
    s = O.score_text_attention(lay, q, k, 1, 1, g["scale"])
    assert np.allclose(s, g["expected_scores"], rtol=1e-14, atol=1e-16), g["derivation"]


def _brute_force_scores(lay, q, k, Hq, Hkv, scale, query_set="text"):
    """Full square causal attention per request via scipy softmax; GQA by np.repeat."""
    out = np.zeros(lay.n_tokens)
    vis_all = lay.visual_mask()
    for r in range(lay.n_requests):
        a, b = int(lay.cu_seqlens[r]), int(lay.cu_seqlens[r + 1])
        Q = synth.bf16_bits_to_f32(q[a:b]).astype(np.float64)          # [T, Hq, d]
        K = synth.bf16_bits_to_f32(k[a:b]).astype(np.float64)          # [T, Hkv, d]
        K = np.repeat(K, Hq // Hkv, axis=1)                            # head h -> kv h // (Hq/Hkv)
        logits = np.einsum("qhd,khd->hqk", Q, K) * scale                # [Hq, T, T]
        mask = np.tril(np.ones((b - a, b - a), dtype=bool))            # key <= query
        logits = np.where(mask[None], logits, -np.inf)
        P = ssp.softmax(logits, axis=-1)
        if query_set == "text":
            rows = ~vis_all[a:b]
        else:  # the request's last token alone
            rows = np.zeros(b - a, dtype=bool)
            rows[-1] = b > a
        nq = rows.sum()
        if nq == 0:
            continue
        s = P[:, rows, :].sum(axis=(0, 1)) / (Hq * nq)
        out[a:b][vis_all[a:b]] = s[vis_all[a:b]]
    return out


@pytest.mark.parametrize("Hq,Hkv", [(4, 2), (4, 4), (6, 2)])
def test_text_attention_matches_full_square_attention(Hq, Hkv):
    wl = synth.make_custom([[("t", 5), ("i", 12), ("t", 3), ("i", 7), ("t", 4)], [("i", 9), ("t", 6)]],
                           hidden=32, n_q_heads=Hq, n_kv_heads=Hkv, head_dim=16, seed=3, parts=("B",))
    scale = wl.softmax_scale
    s = O.score_text_attention(wl.layout, wl.q, wl.k, Hq, Hkv, scale)
    ref = _brute_force_scores(wl.layout, wl.q, wl.k, Hq, Hkv, scale)
    assert np.allclose(s, ref, rtol=1e-12, atol=1e-15)


@pytest.mark.parametrize("Hq,Hkv", [(4, 2), (6, 6)])
def test_last_token_attention_matches_full_square_attention(Hq, Hkv):
    for segs in ([[("t", 5), ("i", 12), ("t", 3), ("i", 7), ("t", 4)], [("i", 9), ("t", 6)]],
                 [[("t", 2), ("i", 11)], [("i", 4)]]):  # requests ending in an image
        wl = synth.make_custom(segs, hidden=32, n_q_heads=Hq, n_kv_heads=Hkv, head_dim=16, seed=4, parts=("B",))
        s = O.score_text_attention(wl.layout, wl.q, wl.k, Hq, Hkv, wl.softmax_scale, query_set="last")
        ref = _brute_force_scores(wl.layout, wl.q, wl.k, Hq, Hkv, wl.softmax_scale, query_set="last")
        assert np.allclose(s, ref, rtol=1e-12, atol=1e-15)


def test_last_token_attention_golden():
    g = _load("text_attention_last.json")
    for case in g["cases"]:
        lay = synth.Layout.from_segments([[(k, n) for k, n in case["layout"]]])
        q = _bits(case["q"]).reshape(-1, 1, 1)
        k = _bits(case["k"]).reshape(-1, 1, 1)
        last = O.score_text_attention(lay, q, k, 1, 1, case["scale"], query_set="last")
        text = O.score_text_attention(lay, q, k, 1, 1, case["scale"], query_set="text")
        assert np.allclose(last, case["expected_last"], rtol=1e-14, atol=1e-16), case["name"]
        assert np.allclose(text, case["expected_text"], rtol=1e-14, atol=1e-16), case["name"]


def test_last_token_mass_is_its_softmax_row():
    # the last token's softmax row sums to one over the request's keys, so the visual
    # scores plus the text keys' probabilities make one, for every head
    wl = synth.make_custom([[("t", 3), ("i", 10), ("t", 2), ("i", 6), ("t", 1)]], n_q_heads=2, n_kv_heads=1,
                           head_dim=16, seed=8, parts=("B",))
    vis = wl.layout.visual_mask()
    total = 0.0
    for h in range(2):
        z, qpos = O.attention_logits(wl.layout, wl.q, wl.k, 0, h, 2, 1, wl.softmax_scale, "last")
        assert qpos.tolist() == [wl.layout.n_tokens - 1]
        P = np.exp(z - O.logsumexp_rows(z)[:, None])[0]
        assert P.sum() == pytest.approx(1.0, abs=1e-13)
        total += P[~vis].sum()
    s = O.score_text_attention(wl.layout, wl.q, wl.k, 2, 1, wl.softmax_scale, query_set="last")
    assert s[vis].sum() + total / 2 == pytest.approx(1.0, abs=1e-13)


def test_tiny_config_matches_full_square_attention():
    wl = synth.make_workload("tiny", parts=("B",))
    s = O.score_text_attention(wl.layout, wl.q, wl.k, 4, 2, wl.softmax_scale)
    ref = _brute_force_scores(wl.layout, wl.q, wl.k, 4, 2, wl.softmax_scale)
    assert np.allclose(s, ref, rtol=1e-12, atol=1e-16)


def test_softmax_rows_sum_to_one():
    wl = synth.make_custom([[("t", 4), ("i", 20), ("t", 6)]], n_q_heads=4, n_kv_heads=2,
                           head_dim=16, seed=5, parts=("B",))
    for h in range(4):
        z, text_local = O.attention_logits(wl.layout, wl.q, wl.k, 0, h, 4, 2, wl.softmax_scale)
        lse = O.logsumexp_rows(z)
        P = np.exp(z - lse[:, None])
        assert np.allclose(P.sum(axis=1), 1.0, atol=1e-13)
        # nothing leaks past the causal frontier
        keys = np.arange(z.shape[1])
        assert np.all(P[keys[None, :] > text_local[:, None]] == 0.0)


def test_zero_queries_give_uniform_attention():
    lay = synth.Layout.from_segments([[("t", 3), ("i", 5), ("t", 2), ("i", 4), ("t", 2)]])
    T, Hq, Hkv, d = lay.n_tokens, 2, 1, 8
    rng = np.random.default_rng(2)
    q = np.zeros((T, Hq, d), dtype=np.uint16)              # bf16 +0
    k = _bits(rng.standard_normal((T * Hkv * d))).reshape(T, Hkv, d)
    s = O.score_text_attention(lay, q, k, Hq, Hkv, 0.25)
    vis = lay.visual_mask()
    text_pos = np.nonzero(~vis)[0]
    for t in np.nonzero(vis)[0]:
        # every text query q >= t spreads 1/(q+1) on each visible key
        expect = sum(1.0 / (p + 1) for p in text_pos if p >= t) / len(text_pos)
        assert s[t] == pytest.approx(expect, rel=1e-14)


def test_single_visible_key_lse():
    lay = synth.Layout.from_segments([[("t", 1), ("i", 3), ("t", 1)]])
    rng = np.random.default_rng(4)
    q = _bits(rng.standard_normal((5 * 2 * 8))).reshape(5, 2, 8)
    k = _bits(rng.standard_normal((5 * 1 * 8))).reshape(5, 1, 8)
    lse = O.text_lse(lay, q, k, 2, 1, 0.5)
    for h in range(2):
        z00 = 0.5 * float(np.dot(synth.bf16_bits_to_f32(q[0, h]).astype(np.float64),
                                 synth.bf16_bits_to_f32(k[0, 0]).astype(np.float64)))
        assert lse[h, 0] == pytest.approx(z00, abs=1e-14)  # log(exp(z)) = z: P = 1


def test_supplied_lse_reproduces_scores():
    wl = synth.make_custom([[("t", 6), ("i", 10), ("t", 2), ("i", 10), ("t", 5)]], seed=9, parts=("B",))
    lse = O.text_lse(wl.layout, wl.q, wl.k, 4, 2, wl.softmax_scale)
    a = O.score_text_attention(wl.layout, wl.q, wl.k, 4, 2, wl.softmax_scale)
    b = O.score_text_attention(wl.layout, wl.q, wl.k, 4, 2, wl.softmax_scale, lse=lse)
    assert np.allclose(a, b, rtol=1e-13, atol=1e-16)
    # a shifted normaliser scales every probability by exp(-shift)
    c = O.score_text_attention(wl.layout, wl.q, wl.k, 4, 2, wl.softmax_scale, lse=lse + math.log(2.0))
    assert np.allclose(c, a / 2.0, rtol=1e-13, atol=1e-16)


def test_request_without_text_scores_zero():
    wl = synth.make_custom([[("i", 8), ("i", 8)]], seed=1, parts=("B",))
    s = O.score_text_attention(wl.layout, wl.q, wl.k, 4, 2, wl.softmax_scale)
    assert np.all(s == 0.0)


# ---------------------------------------------------------------- fixed point
def test_fixed_point_values():
    v = np.array([0.5, -0.25, np.nan, 2048.0, -np.inf, 2.0 ** -33, 3 * 2.0 ** -33, 0.0], dtype=np.float32)
    fx = O.fixed_point(v)
    assert fx.tolist() == [2 ** 31, -(2 ** 30), 0, 2 ** 42, -(2 ** 42), 0, 2, 0]


# ---------------------------------------------------------------- step 2
def _alloc_case(case):
    lay = synth.Layout.from_segments([[(k, n) for k, n in case["layout"]]])
    scores = np.zeros(lay.n_tokens, dtype=np.float32)
    for i, v in enumerate(case["image_scores"]):
        s = int(lay.img_start[i])
        scores[s:s + int(lay.img_len[i])] = v
    S = O.image_sums(lay, scores)
    kr = np.array([case["keep_ratio"]], dtype=np.float32)
    return lay, O.allocate(lay, S, kr, case["alpha"], 0.05, 0.95, case["relative"])


def test_allocation_golden():
    for case in _load("allocation.json")["cases"]:
        lay, res = _alloc_case(case)
        assert res["budgets"].tolist() == case["expected_budgets"], case["name"] + ": " + case["derivation"]
        assert int(res["out_cu_seqlens"][-1]) == case["expected_out_len"], case["name"]


def test_allocation_no_clamp_lambda_is_zero():
    # token-weighted mean => sum_i n_i r_i = r_base N_vis: no shift needed when no clamp binds
    case = _load("allocation.json")["cases"][0]
    lay, res = _alloc_case(case)
    assert abs(res["lam"][0]) < 1e-15
    assert np.allclose(res["ratios"], [0.71875, 0.34375, 0.46875], rtol=0, atol=1e-15)


def test_global_budget_rounding():
    assert O.global_budget(np.float32(0.5), 3) == 2          # 1.5 + 0.5
    assert O.global_budget(np.float32(0.25), 5832) == 1458
    assert O.global_budget(np.float32(0.33), 9600) == 3168  # fp32 0.33 = 0.3300000131...
    assert O.global_budget(np.float32(1.0), 7) == 7
    assert O.global_budget(np.float32(0.125), 0) == 0


def test_allocation_rejects_ratio_outside_clamps_and_oversized_sums():
    # App. A.2: with r_base below r_min (above r_max) every shifted ratio is clamped up
    # (down) and the kept total would exceed (fall short of) the global budget
    lay = synth.Layout.from_segments([[("i", 40), ("t", 3), ("i", 60)]])
    S = np.array([40 * 2 ** 31, 60 * 2 ** 30], dtype=np.int64)
    for kr in (0.0, 0.04, 0.96, 1.0):
        with pytest.raises(ValueError):
            O.allocate(lay, S, np.array([kr], dtype=np.float32), 1.0, 0.05, 0.95)
    for kr in (0.05, 0.95):
        O.allocate(lay, S, np.array([kr], dtype=np.float32), 1.0, 0.05, 0.95)
    with pytest.raises(ValueError):
        O.allocate(lay, np.array([(40 << 42) + 1, 0], dtype=np.int64), np.array([0.5], dtype=np.float32))


def _random_alloc(rng, m, relative=False, alpha=1.0, kr=None):
    n = rng.integers(1, 300, size=m)
    segs = []
    for v in n:
        segs += [("t", int(rng.integers(0, 3))), ("i", int(v))]
    lay = synth.Layout.from_segments([segs])
    S = rng.integers(0, 2 ** 33, size=m).astype(np.int64) * n  # mean in [0, 2)
    kr = np.array([rng.choice([0.05, 0.125, 0.25, 0.33, 0.5, 0.9]) if kr is None else kr], dtype=np.float32)
    return lay, S, kr, O.allocate(lay, S, kr, alpha, 0.05, 0.95, relative)


@pytest.mark.parametrize("relative", [False, True])
def test_allocation_conserves_total_and_bounds(relative):
    rng = np.random.default_rng(11)
    for trial in range(60):
        m = int(rng.integers(1, 20))
        alpha = float(rng.choice([0.0, 1.0, 2.0, 5.0]))
        lay, S, kr, res = _random_alloc(rng, m, relative, alpha)
        n = lay.img_len.astype(np.int64)
        B = O.global_budget(kr[0], int(n.sum()))
        k = res["budgets"].astype(np.int64)
        assert k.sum() == B
        assert np.all(k >= 0) and np.all(k <= n)
        r_min, r_max = float(np.float32(0.05)), float(np.float32(0.95))
        assert np.all(k >= np.floor(r_min * n) - 1)
        assert np.all(k <= np.floor(r_max * n) + 1)
        T_txt = lay.n_tokens - int(n.sum())
        assert int(res["out_cu_seqlens"][-1]) == B + T_txt


def test_allocation_alpha_zero_is_uniform():
    rng = np.random.default_rng(12)
    for trial in range(30):
        lay, S, kr, res = _random_alloc(rng, int(rng.integers(1, 12)), alpha=0.0)
        n = lay.img_len.astype(np.float64)
        target = float(kr[0]) * n * (O.global_budget(kr[0], int(n.sum())) / (float(kr[0]) * n.sum()))
        assert np.all(np.abs(res["budgets"] - target) <= 1.0 + 1e-9)


def test_identical_images_equal_budgets():
    for m, kr in [(4, 0.5), (3, 0.33), (8, 0.125)]:
        lay = synth.Layout.from_segments([[("t", 2)] + [("i", 96)] * m + [("t", 5)]])
        S = np.full(m, 96 * 2 ** 30, dtype=np.int64)
        res = O.allocate(lay, S, np.array([kr], dtype=np.float32), 1.0, 0.05, 0.95, False)
        k = res["budgets"]
        assert k.max() - k.min() <= 1
        assert np.all(np.diff(k) <= 0)  # the extra tokens go to the lower image indices
        B = O.global_budget(np.float32(kr), 96 * m)
        if (B * 96) % (96 * m) == 0:
            assert k.max() == k.min()


def test_budgets_are_permutation_equivariant():
    rng = np.random.default_rng(13)
    for trial in range(25):
        m = int(rng.integers(2, 10))
        n = rng.integers(16, 200, size=m)
        S = (rng.integers(1, 2 ** 32, size=m).astype(np.int64) * n)
        perm = rng.permutation(m)
        lay1 = synth.Layout.from_segments([[("i", int(v)) for v in n] + [("t", 3)]])
        lay2 = synth.Layout.from_segments([[("i", int(v)) for v in n[perm]] + [("t", 3)]])
        kr = np.array([0.3], dtype=np.float32)
        k1 = O.allocate(lay1, S, kr, 1.0)["budgets"]
        k2 = O.allocate(lay2, S[perm], kr, 1.0)["budgets"]
        assert k2.tolist() == k1[perm].tolist()


def test_more_importance_never_fewer_tokens():
    rng = np.random.default_rng(14)
    for trial in range(25):
        m = int(rng.integers(2, 10))
        n = rng.integers(16, 200, size=m)
        S = (rng.integers(1, 2 ** 31, size=m).astype(np.int64) * n)
        lay = synth.Layout.from_segments([[("i", int(v)) for v in n]])
        kr = np.array([0.4], dtype=np.float32)
        k1 = O.allocate(lay, S, kr, 2.0)["budgets"]
        j = int(rng.integers(0, m))
        S2 = S.copy()
        S2[j] += int(n[j]) * 2 ** 29
        k2 = O.allocate(lay, S2, kr, 2.0)["budgets"]
        assert k2[j] >= k1[j]


def test_relative_rule_is_proportional_to_image_mass():
    # alpha = 1, relative: r_i = r_base * Ibar_i / Ibar_avg, so x_i = B * S_i / sum S
    n = np.array([100, 300, 200])
    S = np.array([100 * 2 ** 30, 300 * 2 ** 31, 200 * 3 * 2 ** 29], dtype=np.int64)
    lay = synth.Layout.from_segments([[("i", 100), ("i", 300), ("i", 200)]])
    res = O.allocate(lay, S, np.array([0.5], dtype=np.float32), 1.0, 0.0, 1.0, True)
    B = 300
    x = B * S / S.sum()
    assert np.all(np.abs(res["budgets"] - x) < 1.0)


def test_relative_rule_is_scale_invariant():
    # Ibar_i / Ibar_avg does not change when every score is multiplied by the same
    # positive factor, so neither do the relative rule's budgets; means of ~1e-7 included
    rng = np.random.default_rng(15)
    for trial in range(40):
        m = int(rng.integers(1, 9))
        n = rng.integers(1, 400, size=m)
        lay = synth.Layout.from_segments([[("t", 1)] + [("i", int(v)) for v in n]])
        S = rng.integers(1, 2 ** 12, size=m).astype(np.int64) * n + rng.integers(0, n)
        kr = np.array([rng.choice([0.125, 0.33, 0.5])], dtype=np.float32)
        alpha = float(rng.choice([0.5, 1.0, 3.0]))
        k1 = O.allocate(lay, S, kr, alpha, 0.05, 0.95, True)["budgets"]
        for c in (3, 2 ** 20 + 7):
            k2 = O.allocate(lay, S * c, kr, alpha, 0.05, 0.95, True)["budgets"]
            assert k2.tolist() == k1.tolist(), (trial, c)


def test_additive_rule_ignores_a_common_shift_of_the_means():
    # adding the same c to every image's mean moves every r_i by alpha*c - alpha*c = 0
    rng = np.random.default_rng(16)
    for trial in range(40):
        m = int(rng.integers(1, 9))
        n = rng.integers(1, 400, size=m)
        lay = synth.Layout.from_segments([[("i", int(v)) for v in n] + [("t", 2)]])
        S = rng.integers(0, 2 ** 33, size=m).astype(np.int64) * n + rng.integers(0, n)
        kr = np.array([rng.choice([0.125, 0.33, 0.5, 0.9])], dtype=np.float32)
        alpha = float(rng.choice([0.5, 1.0, 5.0]))
        k1 = O.allocate(lay, S, kr, alpha)["budgets"]
        c = int(rng.integers(-2 ** 31, 2 ** 31))
        k2 = O.allocate(lay, S + c * n, kr, alpha)["budgets"]
        assert k2.tolist() == k1.tolist(), trial


def _bisect_shift(r, n, B, lo_r, hi_r, iters=200):
    # an independent route to the shift: bisection on the clamped total in exact
    # rationals, keeping G(lo) < B <= G(hi)
    from fractions import Fraction as F

    def G(lam):
        return sum(int(n[i]) * min(max(r[i] + lam, lo_r), hi_r) for i in range(len(n)))

    lo, hi = lo_r - max(r) - 1, hi_r - min(r) + 1  # G(lo) = N r_min, G(hi) = N r_max
    for _ in range(iters):
        mid = (lo + hi) / 2
        if G(mid) >= B:
            hi = mid
        else:
            lo = mid
    return lo, hi, G


@pytest.mark.parametrize("relative", [False, True])
def test_shift_restores_the_budget_and_matches_bisection(relative):
    from fractions import Fraction as F
    rng = np.random.default_rng(17)
    r_min, r_max = F(float(np.float32(0.05))), F(float(np.float32(0.95)))
    for trial in range(40):
        m = int(rng.integers(1, 7))
        n = [int(v) for v in rng.integers(1, 300, size=m)]
        S = [int(v) * n[i] + int(rng.integers(0, n[i])) for i, v in enumerate(rng.integers(1, 2 ** 33, size=m))]
        kr = np.float32(rng.choice([0.05, 0.125, 0.33, 0.5, 0.9]))
        alpha = float(rng.choice([1.0, 4.0, 20.0]))  # large alpha: clamps bind
        r = O.adaptive_ratios(S, n, kr, alpha, relative)
        B = O.global_budget(kr, sum(n))
        lam = O.water_fill(r, n, B, r_min, r_max)
        lo, hi, G = _bisect_shift(r, n, B, r_min, r_max)
        N = sum(n)
        if N * r_min < B < N * r_max:
            assert G(lam) == B, trial
            assert lo <= lam <= hi, trial
        x = [n[i] * min(max(r[i] + lam, r_min), r_max) for i in range(m)]
        assert all(n[i] * r_min <= x[i] <= n[i] * r_max for i in range(m))


def test_largest_remainder_is_the_closest_integer_vector():
    # Rounding to integers with a fixed total: the largest-remainder vector minimises
    # sum (k_i - x_i)^2 over every integer vector with sum B and 0 <= k_i <= n_i; among
    # several minimisers (equal remainders) the rule favours the lower index, i.e. the
    # lexicographically largest one. Checked by enumeration.
    from fractions import Fraction as F
    rng = np.random.default_rng(18)
    for trial in range(150):
        m = int(rng.integers(1, 5))
        n = [int(v) for v in rng.integers(1, 6, size=m)]
        den = int(rng.choice([1, 2, 3, 4, 7, 10]))
        # kept masses with sum B (the water-fill's output) or just above it (every image at r_min)
        x = [F(int(rng.integers(0, n[i] * den + 1)), den) for i in range(m)]
        B = math.floor(sum(x))
        if trial % 5 == 0 and B > 0:
            B -= 1
        got = O.integer_budgets(x, n, B)
        best = None
        for k in itertools.product(*[range(v + 1) for v in n]):
            if sum(k) != B:
                continue
            key = (sum((k[i] - x[i]) ** 2 for i in range(m)), tuple(-v for v in k))
            if best is None or key < best[0]:
                best = (key, list(k))
        assert got == best[1], (trial, x, B)


# ---------------------------------------------------------------- pruning-layer selection
def test_layer_selection_golden():
    g = _load("layer_selection.json")
    A = np.asarray(g["A"], dtype=np.int64)
    assert O.layer_ranks(A).tolist() == g["expected_ranks"], g["derivation"]
    rank_sum, R = O.mean_ranks(A)
    assert rank_sum.tolist() == g["expected_rank_sum"]
    assert np.allclose(R, np.asarray(g["expected_rank_sum"]) / 3.0, rtol=0, atol=1e-15)
    for k, top in g["expected_top"].items():
        assert O.select_layers(A, int(k)).tolist() == top, k


def test_layer_ranks_match_scipy_ordinal_ranks():
    # scipy's ordinal ranking of -A breaks ties by position: the lower layer first
    import scipy.stats as sst
    rng = np.random.default_rng(41)
    for trial in range(30):
        N, L = int(rng.integers(1, 6)), int(rng.integers(1, 40))
        A = rng.integers(-5, 6, size=(N, L)).astype(np.int64) * int(rng.integers(1, 2 ** 40))
        ranks = O.layer_ranks(A)
        for i in range(N):
            assert ranks[i].tolist() == sst.rankdata(-A[i], method="ordinal").astype(int).tolist()


def test_layer_selection_invariances():
    rng = np.random.default_rng(42)
    for trial in range(30):
        N, L = int(rng.integers(1, 8)), int(rng.integers(2, 30))
        A = rng.permutation(N * L).reshape(N, L).astype(np.int64) * 7 + 3  # distinct values
        rank_sum, _ = O.mean_ranks(A)
        # the order of the samples does not matter
        assert O.mean_ranks(A[rng.permutation(N)])[0].tolist() == rank_sum.tolist()
        # relabelling the layers relabels the result
        perm = rng.permutation(L)
        assert O.mean_ranks(A[:, perm])[0].tolist() == rank_sum[perm].tolist()
        # scaling one sample's attention by a positive factor changes none of its ranks
        B = A.copy()
        B[int(rng.integers(0, N))] *= 5
        assert O.layer_ranks(B).tolist() == O.layer_ranks(A).tolist()
        # the selected layers have the best mean ranks
        k = int(rng.integers(1, L + 1))
        top = O.select_layers(A, k)
        worst_in = max(rank_sum[top])
        rest = np.setdiff1d(np.arange(L), top)
        assert len(rest) == 0 or worst_in <= min(rank_sum[rest])


def test_layer_attention_sums_the_visual_fixed_point_scores():
    wl = synth.make_custom([[("t", 3), ("i", 10), ("t", 2), ("i", 6)], [("i", 4), ("t", 5)], [("t", 2)]],
                           seed=12, parts=("B",))
    s = O.to_fp32(O.score_text_attention(wl.layout, wl.q, wl.k, 4, 2, wl.softmax_scale))
    A = O.layer_attention(wl.layout, O.image_sums(wl.layout, s))
    fx = O.fixed_point(s)
    vis = wl.layout.visual_mask()
    for r in range(wl.layout.n_requests):
        a, b = int(wl.layout.cu_seqlens[r]), int(wl.layout.cu_seqlens[r + 1])
        assert int(A[r]) == int(fx[a:b][vis[a:b]].sum())
    assert int(A[2]) == 0  # a request without images has no visual attention


# ---------------------------------------------------------------- step 3
def test_selection_golden():
    for case in _load("selection.json")["cases"]:
        lay = synth.Layout.from_segments([[(k, n) for k, n in case["layout"]]])
        sc = np.array([_f(v) for v in case["scores"]], dtype=np.float32)
        kept = O.select(lay, sc, np.array(case["budgets"], dtype=np.int32))
        assert kept.tolist() == case["expected_kept"], case["derivation"]


def _dominates(sa, pa, sb, pb):
    """True iff token a ranks strictly above token b: larger score, or equal score and lower position."""
    na, nb = math.isnan(sa), math.isnan(sb)
    if na and nb:
        return pa < pb
    if na:
        return False
    if nb:
        return True
    return sa > sb or (sa == sb and pa < pb)


def test_selection_brute_force_small():
    rng = np.random.default_rng(21)
    pool = np.array([0.0, -0.0, 0.5, 0.5, 1.0, -1.0, np.nan, np.inf, -np.inf, 0.25], dtype=np.float32)
    for trial in range(120):
        n = int(rng.integers(1, 11))
        sc_img = rng.choice(pool, size=n) if trial % 2 else rng.standard_normal(n).astype(np.float32)
        lay = synth.Layout.from_segments([[("t", 1), ("i", n), ("t", 1)]])
        sc = np.zeros(n + 2, dtype=np.float32)
        sc[1:n + 1] = sc_img
        for kk in range(n + 1):
            kept = O.select(lay, sc, np.array([kk], dtype=np.int32))
            # brute force: the unique k-subset whose every member ranks above every non-member
            winners = []
            for sub in itertools.combinations(range(1, n + 1), kk):
                rest = [t for t in range(1, n + 1) if t not in sub]
                if all(_dominates(float(sc[a]), a, float(sc[b]), b) for a in sub for b in rest):
                    winners.append(sub)
            assert len(winners) == 1
            assert kept.tolist() == sorted([0, n + 1] + list(winners[0]))


def test_selection_structure_on_tiny():
    wl = synth.make_workload("tiny", parts=("A",))
    res = O.prune(wl.layout, keep_ratio=wl.keep_ratio, h_cur=wl.h_cur, h_prior=wl.h_prior)
    kept = res["kept_idx"]
    assert np.all(np.diff(kept) > 0)
    vis = wl.layout.visual_mask()
    assert set(np.nonzero(~vis)[0].tolist()) <= set(kept.tolist())   # text never dropped
    assert len(kept) == int(res["out_cu_seqlens"][-1])
    assert int(res["budgets"].sum()) == O.global_budget(wl.keep_ratio[0], int(vis.sum()))
    # image importance grows with the synthetic signal (0, 0.5, 1): so do the budgets
    assert res["budgets"][0] < res["budgets"][1] < res["budgets"][2]


# ---------------------------------------------------------------- step 4
def test_compact_is_row_gather():
    rng = np.random.default_rng(31)
    rows = rng.integers(0, 2 ** 16, size=(50, 7), dtype=np.uint16)
    planes = rng.integers(0, 2 ** 31, size=(3, 50), dtype=np.int64).astype(np.int32)
    idx = np.array(sorted(rng.choice(50, size=17, replace=False)), dtype=np.int32)
    out = O.compact(idx, rows)
    outp = O.compact_planes(idx, planes)
    for j, t in enumerate(idx):
        assert out[j].tobytes() == rows[t].tobytes()
        for p in range(3):
            assert outp[p, j] == planes[p, t]


# ---------------------------------------------------------------- the pruned layout (progressive pruning)
def test_pruned_layout_golden():
    g = _load("pruned_layout.json")
    lay = synth.Layout(**{k: np.asarray(v, dtype=np.int32) for k, v in g["layout"].items()})
    got = O.pruned_layout(lay, np.asarray(g["kept_idx"]), np.asarray(g["out_cu_seqlens"]))
    for k, v in g["expected"].items():
        assert got[k].tolist() == v, k


def _pruned_case(seed):
    rng = np.random.default_rng(seed)
    reqs = []
    for _ in range(rng.integers(1, 4)):
        segs = []
        for _ in range(rng.integers(1, 6)):
            if rng.random() < 0.6:
                segs.append(("i", int(rng.integers(1, 40))))
            else:
                segs.append(("t", int(rng.integers(1, 9))))
        reqs.append(segs)
    lay = synth.Layout.from_segments(reqs)
    scores = rng.standard_normal(lay.n_tokens).astype(np.float32)
    budgets = np.array([rng.integers(0, n + 1) for n in lay.img_len], dtype=np.int32)
    kept = O.select(lay, scores, budgets)
    vis = lay.visual_mask()
    cu2 = [0]
    for r in range(lay.n_requests):
        a, b = int(lay.cu_seqlens[r]), int(lay.cu_seqlens[r + 1])
        n_txt = int((~vis[a:b]).sum())
        cu2.append(cu2[-1] + n_txt + int(budgets[int(lay.img_cu[r]):int(lay.img_cu[r + 1])].sum()))
    return lay, budgets, kept, np.asarray(cu2, dtype=np.int32)


@pytest.mark.parametrize("seed", range(20))
def test_pruned_layout_closed_form(seed):
    # in request r, image i moves left by the tokens pruned from the request's earlier
    # images, and keeps its budget
    lay, budgets, kept, cu2 = _pruned_case(seed)
    got = O.pruned_layout(lay, kept, cu2)
    for r in range(lay.n_requests):
        dropped = 0
        for i in range(int(lay.img_cu[r]), int(lay.img_cu[r + 1])):
            assert got["img_start"][i] == lay.img_start[i] - dropped
            assert got["img_len"][i] == budgets[i]
            dropped += int(lay.img_len[i]) - int(budgets[i])
    assert got["cu_seqlens"].tolist() == cu2.tolist()


@pytest.mark.parametrize("seed", range(20))
def test_pruned_layout_marks_exactly_the_kept_visual_tokens(seed):
    lay, budgets, kept, cu2 = _pruned_case(seed)
    got = O.pruned_layout(lay, kept, cu2)
    lay2 = synth.Layout(cu_seqlens=got["cu_seqlens"], img_cu=got["img_cu"], img_start=got["img_start"],
                        img_len=got["img_len"])
    # the visual mask of the pruned batch is the gathered visual mask of the original
    assert np.array_equal(lay2.visual_mask(), lay.visual_mask()[kept])


# ---------------------------------------------------------------- the layer's attention forward
def _fwd_workload(Hq=4, Hkv=2, d=16, seed=11):
    segs = [[("t", 3), ("i", 9), ("t", 2), ("i", 5), ("t", 4)], [("i", 7), ("t", 3)], [("t", 1)]]
    return synth.make_custom(segs, hidden=32, n_q_heads=Hq, n_kv_heads=Hkv, head_dim=d, seed=seed,
                             parts=("B", "V"))


@pytest.mark.parametrize("Hq,Hkv", [(4, 2), (3, 3), (6, 1)])
def test_attention_forward_matches_torch_sdpa(Hq, Hkv):
    """The forward against torch's scaled_dot_product_attention in fp64 (a library routine,
    causal per request, GQA by repeating each KV head over its query heads), and the
    normaliser against torch.logsumexp of the masked logits."""
    torch = pytest.importorskip("torch")
    wl = _fwd_workload(Hq, Hkv)
    lay = wl.layout
    out, lse = O.attention_forward(lay, wl.q, wl.k, wl.v, Hq, Hkv, wl.softmax_scale)
    G = Hq // Hkv
    for r in range(lay.n_requests):
        a, b = int(lay.cu_seqlens[r]), int(lay.cu_seqlens[r + 1])
        q = torch.from_numpy(O.bf16_to_f64(wl.q[a:b])).permute(1, 0, 2)  # [Hq, T_r, d]
        k = torch.from_numpy(O.bf16_to_f64(wl.k[a:b])).permute(1, 0, 2).repeat_interleave(G, dim=0)
        v = torch.from_numpy(O.bf16_to_f64(wl.v[a:b])).permute(1, 0, 2).repeat_interleave(G, dim=0)
        ref = torch.nn.functional.scaled_dot_product_attention(q, k, v, is_causal=True, scale=wl.softmax_scale)
        np.testing.assert_allclose(out[a:b].transpose(1, 0, 2), ref.numpy(), rtol=1e-12, atol=1e-12)
        z = wl.softmax_scale * torch.einsum("hqd,hkd->hqk", q, k)
        mask = torch.ones(b - a, b - a, dtype=torch.bool).tril()
        ref_lse = torch.logsumexp(z.masked_fill(~mask, float("-inf")), dim=-1)
        np.testing.assert_allclose(lse[:, a:b], ref_lse.numpy(), rtol=1e-12, atol=1e-12)


def test_attention_forward_closed_forms():
    """A request's first token sees only itself: O = its value, lse = its own logit. With
    all queries zero every visible key weighs the same: O = the prefix mean of the values,
    lse = ln(p + 1)."""
    Ox = O
    wl = _fwd_workload()
    lay = wl.layout
    Hq, Hkv, G = wl.n_q_heads, wl.n_kv_heads, wl.n_q_heads // wl.n_kv_heads
    out, lse = Ox.attention_forward(lay, wl.q, wl.k, wl.v, Hq, Hkv, wl.softmax_scale)
    for r in range(lay.n_requests):
        a = int(lay.cu_seqlens[r])
        for h in range(Hq):
            np.testing.assert_array_equal(out[a, h], Ox.bf16_to_f64(wl.v[a, h // G]))
            z0 = wl.softmax_scale * np.dot(Ox.bf16_to_f64(wl.q[a, h]), Ox.bf16_to_f64(wl.k[a, h // G]))
            assert lse[h, a] == pytest.approx(z0, rel=1e-14, abs=1e-14)
    q0 = np.zeros_like(wl.q)
    out0, lse0 = Ox.attention_forward(lay, q0, wl.k, wl.v, Hq, Hkv, wl.softmax_scale)
    for r in range(lay.n_requests):
        a, b = int(lay.cu_seqlens[r]), int(lay.cu_seqlens[r + 1])
        vf = Ox.bf16_to_f64(wl.v[a:b])                               # [T_r, Hkv, d]
        prefix_mean = np.cumsum(vf, axis=0) / np.arange(1, b - a + 1)[:, None, None]
        for h in range(Hq):
            np.testing.assert_allclose(out0[a:b, h], prefix_mean[:, h // G], rtol=1e-12, atol=1e-13)
            np.testing.assert_allclose(lse0[h, a:b], np.log(np.arange(1, b - a + 1)), rtol=1e-13)


def test_attention_forward_rows_match_the_whole_forward():
    Ox = O
    wl = _fwd_workload()
    lay = wl.layout
    out, lse = Ox.attention_forward(lay, wl.q, wl.k, wl.v, wl.n_q_heads, wl.n_kv_heads, wl.softmax_scale)
    a = int(lay.cu_seqlens[0])
    rows = [0, 4, 11, 22]
    o_r, l_r = Ox.attention_forward_rows(lay, wl.q, wl.k, wl.v, wl.n_q_heads, wl.n_kv_heads, wl.softmax_scale, 0, rows)
    np.testing.assert_allclose(o_r, out[[a + p for p in rows]], rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(l_r, lse[:, [a + p for p in rows]], rtol=1e-13)


def test_forward_normaliser_is_criterion_b_normaliser():
    """The forward's normaliser at the text rows is the one criterion B divides by: the
    text-query scores computed with it (supplied) equal the scores computed from scratch."""
    Ox = O
    wl = _fwd_workload()
    lay = wl.layout
    _, lse = Ox.attention_forward(lay, wl.q, wl.k, wl.v, wl.n_q_heads, wl.n_kv_heads, wl.softmax_scale)
    s_own = Ox.score_text_attention(lay, wl.q, wl.k, wl.n_q_heads, wl.n_kv_heads, wl.softmax_scale)
    s_fwd = Ox.score_text_attention(lay, wl.q, wl.k, wl.n_q_heads, wl.n_kv_heads, wl.softmax_scale, lse=lse)
    np.testing.assert_allclose(s_fwd, s_own, rtol=1e-12, atol=1e-15)
