"""GPU parity: every step of the pruning stage, through the C ABI, against the fp64 oracle.

Scores: rel 1e-3 / abs 1e-5 (bf16 inputs, fp32 accumulation). Budgets, kept
indices and compacted rows: bit-exact when both sides are fed the same fp32
scores. End to end, index sets may differ only at near-ties of the oracle's
scores.
"""
import numpy as np
import pytest
import torch

from oracle import avtp_oracle as O
from paper_2608_26806_gb300 import avtp, synth
from tests.gpu_util import (ATOL, RTOL, DevWorkload, assert_scores_close, bits_of, dev_layout, ensure_built,
                            near_tie)

pytestmark = pytest.mark.gpu

CONFIGS = ["tiny", "llava_ov_7b", "qwen3_vl_8b", "internvl3_5_8b"]


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    ensure_built()


_CACHE = {}


def workload(name):
    if name not in _CACHE:
        wl = synth.make_workload(name)
        _CACHE.clear()  # keep one large workload resident at a time
        _CACHE[name] = (wl, DevWorkload(wl))
    return _CACHE[name]


def oracle_scores(wl, criterion):
    if criterion == "hidden_variation":
        return O.score_hidden_variation(wl.layout, wl.h_cur, wl.h_prior)
    return O.score_text_attention(wl.layout, wl.q, wl.k, wl.n_q_heads, wl.n_kv_heads, wl.softmax_scale)


# ---------------------------------------------------------------- step 1
@pytest.mark.parametrize("name", CONFIGS)
@pytest.mark.parametrize("criterion", ["hidden_variation", "text_attention"])
def test_score_parity(name, criterion):
    wl, dw = workload(name)
    scores, sums = avtp.score(dw.L, criterion, **dw.score_tensors(criterion))
    torch.cuda.synchronize()
    got = scores.cpu().numpy()
    ref = oracle_scores(wl, criterion)
    vis = wl.layout.visual_mask()
    assert_scores_close(got, ref, vis)
    # the fixed-point per-image sums of the GPU's own scores are exact integers
    assert np.array_equal(sums.cpu().numpy(), O.image_sums(wl.layout, got))


@pytest.mark.parametrize("name", ["tiny", "qwen3_vl_8b"])
def test_score_attention_with_supplied_lse(name):
    wl, dw = workload(name)
    lse = O.text_lse(wl.layout, wl.q, wl.k, wl.n_q_heads, wl.n_kv_heads, wl.softmax_scale)
    lse_dev = torch.from_numpy(lse.astype(np.float32)).cuda()
    scores, _ = avtp.score(dw.L, "text_attention", lse=lse_dev, **dw.score_tensors("text_attention"))
    torch.cuda.synchronize()
    ref = O.score_text_attention(wl.layout, wl.q, wl.k, wl.n_q_heads, wl.n_kv_heads, wl.softmax_scale,
                                 lse=lse.astype(np.float32).astype(np.float64))
    assert_scores_close(scores.cpu().numpy(), ref, wl.layout.visual_mask())


# Layouts that stress the text-attention bookkeeping: row blocks of 256 (query, head)
# rows that end mid-request or hold one row, requests without text or without images,
# text only before the images, adjacent images, images of 1 and of 129 tokens, and
# several blocks and key steps per request.
_ATTN_EDGE_LAYOUTS = [
    [[("i", 40), ("t", 3), ("i", 300), ("t", 100)], [("t", 5)], [("i", 17)],
     [("t", 70), ("i", 129), ("i", 1), ("t", 1)]],
    [[("t", 1), ("i", 256), ("t", 1)], [("i", 5), ("t", 200), ("i", 300), ("t", 9)]],
    [[("t", 65), ("i", 10), ("t", 64), ("i", 7), ("t", 1)], [("t", 30), ("i", 600)]],
    [[("t", 300), ("i", 513), ("t", 2), ("i", 700), ("t", 140)]],
]


@pytest.mark.parametrize("layout_id", range(len(_ATTN_EDGE_LAYOUTS)))
@pytest.mark.parametrize("heads", [(4, 4, 64), (6, 2, 64), (12, 4, 128), (7, 1, 128)])
@pytest.mark.parametrize("supplied_lse", [False, True])
def test_score_attention_edge_layouts(layout_id, heads, supplied_lse):
    Hq, Hkv, d = heads
    wl = synth.make_custom(_ATTN_EDGE_LAYOUTS[layout_id], n_q_heads=Hq, n_kv_heads=Hkv, head_dim=d, hidden=64,
                           seed=11 + layout_id, parts=("B",))
    dw = DevWorkload(wl)
    kw = {}
    ref_lse = None
    if supplied_lse:
        lse = O.text_lse(wl.layout, wl.q, wl.k, Hq, Hkv, wl.softmax_scale)
        kw["lse"] = torch.from_numpy(lse.astype(np.float32)).cuda()
        ref_lse = lse.astype(np.float32).astype(np.float64)
    scores, sums = avtp.score(dw.L, "text_attention", **kw, **dw.score_tensors("text_attention"))
    torch.cuda.synchronize()
    got = scores.cpu().numpy()
    ref = O.score_text_attention(wl.layout, wl.q, wl.k, Hq, Hkv, wl.softmax_scale, lse=ref_lse)
    vis = wl.layout.visual_mask()
    assert_scores_close(got, ref, vis)
    assert np.array_equal(sums.cpu().numpy(), O.image_sums(wl.layout, got))


# ---------------------------------------------------------------- step 1B: query sets and paths
@pytest.mark.parametrize("name", CONFIGS)
def test_score_last_token_parity(name):
    # the request's last token as the only query (the output token's attention, §4.1),
    # on the CUDA-core path that query set always takes
    wl, dw = workload(name)
    scores, sums = avtp.score(dw.L, "text_attention", query_set="last", **dw.score_tensors("text_attention"))
    torch.cuda.synchronize()
    got = scores.cpu().numpy()
    ref = O.score_text_attention(wl.layout, wl.q, wl.k, wl.n_q_heads, wl.n_kv_heads, wl.softmax_scale,
                                 query_set="last")
    assert_scores_close(got, ref, wl.layout.visual_mask())
    assert np.array_equal(sums.cpu().numpy(), O.image_sums(wl.layout, got))


@pytest.mark.parametrize("path", ["tensor", "cuda"])
@pytest.mark.parametrize("supplied_lse", [False, True])
def test_score_text_attention_both_paths_on_tiny(path, supplied_lse):
    wl, dw = workload("tiny")
    kw, ref_lse = {}, None
    if supplied_lse:
        lse = O.text_lse(wl.layout, wl.q, wl.k, wl.n_q_heads, wl.n_kv_heads, wl.softmax_scale)
        kw["lse"] = torch.from_numpy(lse.astype(np.float32)).cuda()
        ref_lse = lse.astype(np.float32).astype(np.float64)
    scores, sums = avtp.score(dw.L, "text_attention", path=path, **kw, **dw.score_tensors("text_attention"))
    torch.cuda.synchronize()
    got = scores.cpu().numpy()
    ref = O.score_text_attention(wl.layout, wl.q, wl.k, wl.n_q_heads, wl.n_kv_heads, wl.softmax_scale, lse=ref_lse)
    assert_scores_close(got, ref, wl.layout.visual_mask())
    assert np.array_equal(sums.cpu().numpy(), O.image_sums(wl.layout, got))


@pytest.mark.parametrize("layout_id", range(len(_ATTN_EDGE_LAYOUTS)))
@pytest.mark.parametrize("heads", [(4, 4, 64), (6, 2, 64), (12, 4, 128), (7, 1, 128)])
@pytest.mark.parametrize("query_set", ["text", "last"])
@pytest.mark.parametrize("supplied_lse", [False, True])
def test_score_cuda_core_path_edge_layouts(layout_id, heads, query_set, supplied_lse):
    Hq, Hkv, d = heads
    wl = synth.make_custom(_ATTN_EDGE_LAYOUTS[layout_id], n_q_heads=Hq, n_kv_heads=Hkv, head_dim=d, hidden=64,
                           seed=11 + layout_id, parts=("B",))
    dw = DevWorkload(wl)
    kw, ref_lse = {}, None
    if supplied_lse:
        lse = O.text_lse(wl.layout, wl.q, wl.k, Hq, Hkv, wl.softmax_scale, query_set=query_set)
        kw["lse"] = torch.from_numpy(lse.astype(np.float32)).cuda()
        ref_lse = lse.astype(np.float32).astype(np.float64)
    scores, sums = avtp.score(dw.L, "text_attention", path="cuda", query_set=query_set, **kw,
                              **dw.score_tensors("text_attention"))
    torch.cuda.synchronize()
    got = scores.cpu().numpy()
    ref = O.score_text_attention(wl.layout, wl.q, wl.k, Hq, Hkv, wl.softmax_scale, lse=ref_lse, query_set=query_set)
    assert_scores_close(got, ref, wl.layout.visual_mask())
    assert np.array_equal(sums.cpu().numpy(), O.image_sums(wl.layout, got))


def test_prune_last_token_end_to_end():
    wl, dw = workload("qwen3_vl_8b")
    out = avtp.prune(dw.L, "text_attention", keep_ratio=dw.keep_ratio, keep_ratio_host=wl.keep_ratio,
                     rows={"hidden": dw.t["h_cur"]}, planes={"pos": dw.t["pos"]}, query_set="last",
                     **dw.score_tensors("text_attention"))
    torch.cuda.synchronize()
    assert avtp.read_device_status(out.workspace) == avtp.OK
    got = out.scores.cpu().numpy()
    ref64 = O.score_text_attention(wl.layout, wl.q, wl.k, wl.n_q_heads, wl.n_kv_heads, wl.softmax_scale,
                                   query_set="last")
    assert_scores_close(got, ref64, wl.layout.visual_mask())
    ref = O.prune(wl.layout, keep_ratio=wl.keep_ratio, scores_f32=got, relative=True, rows={"hidden": wl.h_cur},
                  planes={"pos": wl.pos})
    assert np.array_equal(out.budgets[:wl.layout.n_images].cpu().numpy(), ref["budgets"])
    assert np.array_equal(out.kept_idx.cpu().numpy(), ref["kept_idx"])
    assert np.array_equal(bits_of(out.outputs["hidden"]), ref["hidden"])


def test_tensor_path_rejects_the_last_token_set():
    wl, dw = workload("tiny")
    with pytest.raises(avtp.AVTPError) as e:
        avtp.score(dw.L, "text_attention", path="tensor", query_set="last", **dw.score_tensors("text_attention"))
    assert e.value.code == avtp.ERR_UNSUPPORTED


# ---------------------------------------------------------------- step 2
@pytest.mark.parametrize("name", CONFIGS)
@pytest.mark.parametrize("relative", [False, True])
def test_allocate_bit_exact_on_oracle_sums(name, relative):
    wl, dw = workload(name)
    crit = "text_attention" if relative else "hidden_variation"
    s32 = O.to_fp32(oracle_scores(wl, crit))
    S = O.image_sums(wl.layout, s32)
    ref = O.allocate(wl.layout, S, wl.keep_ratio, 1.0, 0.05, 0.95, relative)
    budgets, out_cu = avtp.allocate(dw.L, torch.from_numpy(S).cuda(), dw.keep_ratio, 1.0, 0.05, 0.95, relative)
    torch.cuda.synchronize()
    assert np.array_equal(budgets.cpu().numpy(), ref["budgets"])
    assert np.array_equal(out_cu.cpu().numpy(), ref["out_cu_seqlens"])


def test_allocate_bit_exact_random_strong_signal():
    rng = np.random.default_rng(7)
    for trial in range(40):
        R = int(rng.integers(1, 5))
        reqs = []
        for _ in range(R):
            segs = [("t", int(rng.integers(0, 5)))]
            for _ in range(int(rng.integers(0, 40))):
                segs += [("i", int(rng.integers(1, 700))), ("t", int(rng.integers(0, 3)))]
            reqs.append(segs)
        lay = synth.Layout.from_segments(reqs)
        n = lay.img_len.astype(np.int64)
        S = (rng.integers(-2 ** 33, 2 ** 34, size=lay.n_images) * n).astype(np.int64)
        r_min, r_max = (0.05, 0.95) if trial % 3 else (0.0, 1.0)
        choices = [0.05, 0.125, 0.25, 0.33, 0.5, 0.9] + ([0.95] if trial % 3 else [0.0, 1.0])
        kr = rng.choice(np.array(choices, dtype=np.float32), size=R)
        alpha = float(rng.choice([0.0, 1.0, 2.0, 5.0, 100.0]))
        relative = bool(trial % 2)
        ref = O.allocate(lay, S, kr, alpha, r_min, r_max, relative)
        L = dev_layout(lay)
        budgets, out_cu = avtp.allocate(L, torch.from_numpy(S).cuda(), torch.from_numpy(kr).cuda(), alpha, r_min,
                                        r_max, relative)
        torch.cuda.synchronize()
        assert np.array_equal(budgets.cpu().numpy(), ref["budgets"]), trial
        assert np.array_equal(out_cu.cpu().numpy(), ref["out_cu_seqlens"]), trial
        assert avtp.kept_count_host(L.host, kr) == int(ref["out_cu_seqlens"][-1])


def test_allocate_bit_exact_extreme_sums_and_alphas():
    # sums at the +-n * 2^42 bound, means of either sign, zero or of a few 2^-32 units,
    # alpha from the smallest multiple of 2^-32 used here to the 1024 limit, both rules:
    # the budgets must equal the exact rule's to the bit
    rng = np.random.default_rng(8)
    alphas = [0.0, 2.0 ** -32, 2.0 ** -20, 0.3, 1.0, 37.5, 1024.0]
    for trial in range(42):
        R = int(rng.integers(1, 4))
        reqs = [[("t", 2)] + [("i", int(rng.integers(1, 3000))) for _ in range(int(rng.integers(1, 45)))]
                for _ in range(R)]
        lay = synth.Layout.from_segments(reqs)
        n = lay.img_len.astype(np.int64)
        kind = trial % 6
        if kind == 0:
            S = rng.choice([-1, 1], size=lay.n_images) * (n << 42)
        elif kind == 1:
            S = -(rng.integers(0, 2 ** 33, size=lay.n_images) * n)
        elif kind == 2:
            S = np.zeros(lay.n_images, dtype=np.int64)
        elif kind == 3:
            S = rng.integers(-2 ** 20, 2 ** 20, size=lay.n_images)  # means of a few 2^-32 units
        else:
            S = rng.integers(0, 2 ** 34, size=lay.n_images) * n + rng.integers(-n, n + 1)
        S = np.asarray(S, dtype=np.int64)
        r_min, r_max = (0.0, 1.0) if trial % 2 else (0.05, 0.95)
        kr = rng.choice(np.array([r_min, 0.05, 0.33, 0.5, r_max], dtype=np.float32), size=R)
        alpha = alphas[trial % len(alphas)]
        relative = bool((trial // 6) % 2)
        ref = O.allocate(lay, S, kr, alpha, r_min, r_max, relative)
        L = dev_layout(lay)
        budgets, out_cu = avtp.allocate(L, torch.from_numpy(S).cuda(), torch.from_numpy(kr).cuda(), alpha, r_min,
                                        r_max, relative)
        torch.cuda.synchronize()
        assert np.array_equal(budgets.cpu().numpy(), ref["budgets"]), trial
        assert np.array_equal(out_cu.cpu().numpy(), ref["out_cu_seqlens"]), trial


def test_allocate_rejects_sums_beyond_bound():
    L = avtp.Layout.from_host([0, 30], [0, 2], [0, 12], [10, 10])
    kr = torch.tensor([0.5], device="cuda")
    for bad in ([(10 << 42) + 1, 0], [0, -(10 << 42) - 1]):
        sums = torch.tensor(bad, dtype=torch.int64, device="cuda")
        st = _status_after(lambda ws: avtp.allocate(L, sums, kr, workspace=ws))
        assert st == avtp.ERR_DEVICE_INPUT
    with pytest.raises(ValueError):
        O.allocate(synth.Layout.from_segments([[("i", 10), ("t", 2), ("i", 10)]]),
                   np.array([(10 << 42) + 1, 0], dtype=np.int64), np.array([0.5], dtype=np.float32))


def test_allocate_exact_where_a_grid_would_round():
    # Means of a few hundred 2^-32 units under the relative rule, where ratios rounded on a
    # fixed grid move budgets by a token, and large alpha with many clamped images, where
    # the partition the grid's shift implies can be wrong near a breakpoint and the exact
    # search over the breakpoints decides. Requests of up to 70 images take both the
    # register path (<= 32 images) and the shared-memory path of the kernels.
    rng = np.random.default_rng(31)
    for trial in range(48):
        R = int(rng.integers(1, 4))
        reqs = []
        for _ in range(R):
            m = int(rng.choice([1, 2, 3, 7, 16, 31, 32, 33, 50, 70]))
            reqs.append([("t", 1)] + [("i", int(rng.integers(1, 900))) for _ in range(m)])
        lay = synth.Layout.from_segments(reqs)
        n = lay.img_len.astype(np.int64)
        kind = trial % 4
        if kind == 0:
            S = rng.integers(100, 1000, size=lay.n_images) * n + rng.integers(0, n)       # means ~1e-7
        elif kind == 1:
            S = rng.integers(1, 64, size=lay.n_images).astype(np.int64)                    # means < 1 unit
        elif kind == 2:
            S = rng.integers(0, 2 ** 33, size=lay.n_images) * n                            # means in [0, 2)
        else:
            S = np.repeat(rng.integers(1, 2 ** 20, size=1), lay.n_images) * n              # identical means
        S = np.asarray(S, dtype=np.int64)
        alpha = float(rng.choice([1.0, 4.0, 64.0, 1024.0]))
        relative = bool(rng.integers(0, 2)) if kind != 0 else True
        kr = rng.choice(np.array([0.05, 0.125, 0.33, 0.5, 0.95], dtype=np.float32), size=R)
        ref = O.allocate(lay, S, kr, alpha, 0.05, 0.95, relative)
        L = dev_layout(lay)
        budgets, out_cu = avtp.allocate(L, torch.from_numpy(S).cuda(), torch.from_numpy(kr).cuda(), alpha, 0.05,
                                        0.95, relative)
        torch.cuda.synchronize()
        assert np.array_equal(budgets.cpu().numpy(), ref["budgets"]), (trial, kind, alpha, relative)
        assert np.array_equal(out_cu.cpu().numpy(), ref["out_cu_seqlens"]), trial


def test_allocate_golden_cases_on_the_device():
    # the hand-derived cases of tests/golden/allocation.json, through the C ABI
    import json
    import os
    with open(os.path.join(os.path.dirname(__file__), "golden", "allocation.json")) as f:
        cases = json.load(f)["cases"]
    for case in cases:
        lay = synth.Layout.from_segments([[(k, n) for k, n in case["layout"]]])
        scores = np.zeros(lay.n_tokens, dtype=np.float32)
        for i, v in enumerate(case["image_scores"]):
            s = int(lay.img_start[i])
            scores[s:s + int(lay.img_len[i])] = v
        S = O.image_sums(lay, scores)
        L = dev_layout(lay)
        kr = torch.tensor([case["keep_ratio"]], dtype=torch.float32, device="cuda")
        budgets, out_cu = avtp.allocate(L, torch.from_numpy(S).cuda(), kr, case["alpha"], 0.05, 0.95,
                                        case["relative"])
        torch.cuda.synchronize()
        assert budgets.cpu().numpy().tolist() == case["expected_budgets"], case["name"]
        assert int(out_cu[-1]) == case["expected_out_len"], case["name"]


def test_allocate_parameters_outside_the_exact_domain():
    # alpha and the clamps must be multiples of 2^-32 (host check), and so must every keep
    # ratio (device check)
    L = avtp.Layout.from_host([0, 30], [0, 2], [0, 12], [10, 10])
    sums = torch.tensor([10 << 30, 10 << 31], dtype=torch.int64, device="cuda")
    kr = torch.tensor([0.5], device="cuda")
    for kw in (dict(alpha=1e-7), dict(alpha=2.0 ** -33), dict(r_min=1e-12, r_max=0.95)):
        with pytest.raises(avtp.AVTPError) as e:
            avtp.allocate(L, sums, kr, **kw)
        assert e.value.code == avtp.ERR_RANGE, kw
    st = _status_after(lambda ws: avtp.allocate(L, sums, torch.tensor([3e-10], device="cuda"), r_min=0.0,
                                                workspace=ws))
    assert st == avtp.ERR_DEVICE_INPUT
    st = _status_after(lambda ws: avtp.allocate(L, sums, torch.tensor([2.0 ** -30], device="cuda"), r_min=0.0,
                                                workspace=ws))
    assert st == avtp.OK


@pytest.mark.parametrize("alpha", [0.0, 2.0 ** -20, 0.3, 5.0, 1024.0])
@pytest.mark.parametrize("relative", [False, True])
def test_prune_fused_budget_rule_across_alphas(alpha, relative):
    # requests of <= 32 images take the register path of the fused kernel, larger ones
    # the shared-memory path; both must equal the oracle fed the same scores
    rng = np.random.default_rng(9)
    reqs = []
    for m in (1, 5, 32, 33, 70):
        segs = [("t", 3)]
        for _ in range(m):
            segs += [("i", int(rng.integers(1, 120))), ("t", int(rng.integers(0, 2)))]
        reqs.append(segs)
    wl = synth.make_custom(reqs, keep_ratio=0.3, parts=("A", "pos"))
    dw = DevWorkload(wl)
    out = avtp.prune(dw.L, "hidden_variation", keep_ratio=dw.keep_ratio, keep_ratio_host=wl.keep_ratio,
                     alpha=alpha, relative=relative, planes={"pos": dw.t["pos"]},
                     **dw.score_tensors("hidden_variation"))
    torch.cuda.synchronize()
    assert avtp.read_device_status(out.workspace) == avtp.OK
    got = out.scores.cpu().numpy()
    ref = O.prune(wl.layout, keep_ratio=wl.keep_ratio, scores_f32=got, alpha=alpha, relative=relative,
                  planes={"pos": wl.pos})
    assert np.array_equal(out.budgets[:wl.layout.n_images].cpu().numpy(), ref["budgets"])
    assert np.array_equal(out.kept_idx.cpu().numpy(), ref["kept_idx"])


# batches at the edge of the layout rules: no image at all, nothing visual kept (an
# empty output), a one-token image, and a mix of them
_DEGENERATE = {
    "text_only": ([[("t", 7)], [("t", 3)]], 0.5),
    "keep_no_visual": ([[("i", 5)], [("i", 3)]], 0.05),
    "single_token": ([[("i", 1)]], 0.95),
    "mixed": ([[("t", 4)], [("i", 1), ("t", 2)], [("i", 6)]], 0.05),
}


@pytest.mark.parametrize("case", sorted(_DEGENERATE))
@pytest.mark.parametrize("criterion", ["hidden_variation", "text_attention"])
def test_prune_degenerate_batches(case, criterion):
    segs, kr = _DEGENERATE[case]
    wl = synth.make_custom(segs, keep_ratio=kr, parts=("A", "B", "pos"))
    dw = DevWorkload(wl)
    relative = criterion == "text_attention"
    out = avtp.prune(dw.L, criterion, keep_ratio=dw.keep_ratio, keep_ratio_host=wl.keep_ratio,
                     rows={"hidden": dw.t["h_cur"]}, planes={"pos": dw.t["pos"]}, **dw.score_tensors(criterion))
    torch.cuda.synchronize()
    assert avtp.read_device_status(out.workspace) == avtp.OK
    lay = wl.layout
    got = out.scores.cpu().numpy()
    assert_scores_close(got, oracle_scores(wl, criterion), lay.visual_mask())
    ref = O.prune(lay, keep_ratio=wl.keep_ratio, scores_f32=got, relative=relative,
                  rows={"hidden": wl.h_cur}, planes={"pos": wl.pos})
    assert out.n_kept == len(ref["kept_idx"])
    assert np.array_equal(out.budgets[:lay.n_images].cpu().numpy(), ref["budgets"])
    assert np.array_equal(out.out_cu_seqlens.cpu().numpy(), ref["out_cu_seqlens"])
    assert np.array_equal(out.kept_idx[:out.n_kept].cpu().numpy(), ref["kept_idx"])
    assert np.array_equal(bits_of(out.outputs["hidden"]), ref["hidden"])
    assert np.array_equal(out.outputs["pos"].cpu().numpy(), ref["pos"])


# ---------------------------------------------------------------- step 3
def _select_case(lay, scores_f32, budgets):
    L = dev_layout(lay)
    out_cu = np.zeros(lay.n_requests + 1, dtype=np.int32)
    vis = lay.visual_mask()
    for r in range(lay.n_requests):
        a, b = int(lay.cu_seqlens[r]), int(lay.cu_seqlens[r + 1])
        kk = int(budgets[int(lay.img_cu[r]):int(lay.img_cu[r + 1])].sum())
        out_cu[r + 1] = out_cu[r] + kk + int((~vis[a:b]).sum())
    n_kept = int(out_cu[-1])
    kept = avtp.select(L, torch.from_numpy(scores_f32).cuda(), torch.from_numpy(budgets.astype(np.int32)).cuda(),
                       torch.from_numpy(out_cu).cuda(), n_kept)
    torch.cuda.synchronize()
    return kept.cpu().numpy()


@pytest.mark.parametrize("name", CONFIGS)
def test_select_bit_exact_on_oracle_scores(name):
    wl, dw = workload(name)
    s32 = O.to_fp32(oracle_scores(wl, "hidden_variation"))
    ref = O.prune(wl.layout, keep_ratio=wl.keep_ratio, scores_f32=s32)
    got = _select_case(wl.layout, s32, ref["budgets"])
    assert np.array_equal(got, ref["kept_idx"])


def test_select_edge_cases():
    rng = np.random.default_rng(3)
    pool = np.array([0.0, -0.0, 0.5, 0.5, 1.0, -1.0, np.nan, np.inf, -np.inf, 0.25], dtype=np.float32)
    layouts = [
        [[("i", 1), ("t", 2), ("i", 1)]],
        [[("t", 7)], [("i", 5)], [("t", 3), ("i", 9)]],                 # request without images / without text
        [[("i", 3000), ("t", 1), ("i", 1025), ("i", 1024)]],             # multi-tile images
        [[("t", 2), ("i", 40), ("t", 5), ("i", 64)]] * 3,
        [[("i", 2048)]],
    ]
    for li, segs in enumerate(layouts):
        lay = synth.Layout.from_segments(segs)
        for trial in range(6):
            T = lay.n_tokens
            if trial % 3 == 0:
                sc = rng.choice(pool, size=T).astype(np.float32)            # heavy ties, NaN, inf
            elif trial % 3 == 1:
                sc = np.full(T, 0.25, dtype=np.float32)                        # all equal
            else:
                sc = rng.standard_normal(T).astype(np.float32)
            n = lay.img_len
            budgets = np.array([int(rng.integers(0, v + 1)) for v in n], dtype=np.int32)
            if trial == 0:
                budgets = n.copy()           # keep everything
            if trial == 1:
                budgets[:] = 0               # keep text only
            ref = O.select(lay, sc, budgets)
            got = _select_case(lay, sc, budgets)
            assert np.array_equal(got, ref), (li, trial)


# ---------------------------------------------------------------- step 4
@pytest.mark.parametrize("row_shape,dtype", [((4096,), torch.bfloat16), ((8, 128), torch.bfloat16),
                                             ((3,), torch.int16), ((5,), torch.uint8), ((1,), torch.int64),
                                             ((24,), torch.float32)])
def test_compact_bit_exact(row_shape, dtype):
    g = torch.Generator().manual_seed(5)
    T = 3001
    if dtype.is_floating_point:
        src = torch.randn((T,) + row_shape, generator=g).to(dtype)
    else:
        src = torch.randint(0, 100, (T,) + row_shape, generator=g).to(dtype)
    idx = np.sort(np.random.default_rng(1).choice(T, size=1234, replace=False)).astype(np.int32)
    src_d = src.cuda()
    out_d = torch.empty((len(idx),) + row_shape, dtype=dtype, device="cuda")
    avtp.compact(torch.from_numpy(idx).cuda(), T, [(src_d, out_d)])
    torch.cuda.synchronize()
    assert torch.equal(out_d.cpu(), src[torch.from_numpy(idx).long()])


def test_compact_planes_and_strided_rows():
    T = 777
    pos = torch.arange(3 * T, dtype=torch.int32).reshape(3, T)
    big = torch.randn(T, 3 * 256).to(torch.bfloat16)
    view = big[:, 256:512]  # row stride 768 elements, row 256 elements
    idx = torch.arange(0, T, 3, dtype=torch.int32)
    pos_d, view_d = pos.cuda(), big.cuda()[:, 256:512]
    out_pos = torch.empty((3, len(idx)), dtype=torch.int32, device="cuda")
    out_v = torch.empty((len(idx), 256), dtype=torch.bfloat16, device="cuda")
    avtp.compact(idx.cuda(), T, [(view_d, out_v)] + [(pos_d[p], out_pos[p]) for p in range(3)])
    torch.cuda.synchronize()
    assert torch.equal(out_v.cpu(), view[idx.long()])
    assert torch.equal(out_pos.cpu(), pos[:, idx.long()])


# ---------------------------------------------------------------- fused stage
@pytest.mark.parametrize("name", CONFIGS)
@pytest.mark.parametrize("criterion", ["hidden_variation", "text_attention"])
def test_prune_end_to_end(name, criterion):
    wl, dw = workload(name)
    relative = criterion == "text_attention"
    out = avtp.prune(dw.L, criterion, keep_ratio=dw.keep_ratio, keep_ratio_host=wl.keep_ratio,
                     rows={"hidden": dw.t["h_cur"]}, planes={"pos": dw.t["pos"]}, **dw.score_tensors(criterion))
    torch.cuda.synchronize()
    assert avtp.read_device_status(out.workspace) == avtp.OK
    vis = wl.layout.visual_mask()
    got_scores = out.scores.cpu().numpy()
    ref64 = oracle_scores(wl, criterion)
    assert_scores_close(got_scores, ref64, vis)
    # steps 2-4 fed the GPU's own scores: bit-exact
    ref = O.prune(wl.layout, keep_ratio=wl.keep_ratio, scores_f32=got_scores, relative=relative,
                  rows={"hidden": wl.h_cur}, planes={"pos": wl.pos})
    assert np.array_equal(out.img_sums[:wl.layout.n_images].cpu().numpy(), ref["img_sums"])
    assert np.array_equal(out.budgets[:wl.layout.n_images].cpu().numpy(), ref["budgets"])
    assert np.array_equal(out.out_cu_seqlens.cpu().numpy(), ref["out_cu_seqlens"])
    assert np.array_equal(out.kept_idx.cpu().numpy(), ref["kept_idx"])
    assert np.array_equal(bits_of(out.outputs["hidden"]), ref["hidden"])
    assert np.array_equal(out.outputs["pos"].cpu().numpy(), ref["pos"])
    # against the oracle end to end
    _check_against_oracle_end_to_end(wl, got_scores, ref64, ref, relative)


def _check_against_oracle_end_to_end(wl, got_scores, ref64, ref, relative):
    """The GPU's budgets and kept sets against the oracle's own run (its fp64 scores rounded
    to fp32). Budgets may differ only through per-image sums that differ by what the score
    tolerance allows; kept sets only at near-ties of the oracle's scores."""
    lay = wl.layout
    s_ref = O.to_fp32(ref64)
    own = O.prune(lay, keep_ratio=wl.keep_ratio, scores_f32=s_ref, relative=relative)
    assert int(own["out_cu_seqlens"][-1]) == int(ref["out_cu_seqlens"][-1])
    # every image's fixed-point sum within the tolerance the scores are held to
    # (plus one unit of fixed-point rounding per token)
    tol = (ATOL + RTOL * np.abs(s_ref.astype(np.float64))) * 2.0 ** 32 + 1.0
    for i in range(lay.n_images):
        r = int(np.searchsorted(lay.img_cu, i, side="right")) - 1
        s = int(lay.cu_seqlens[r]) + int(lay.img_start[i])
        rows = slice(s, s + int(lay.img_len[i]))
        assert abs(int(ref["img_sums"][i]) - int(own["img_sums"][i])) <= float(tol[rows].sum()), i
    # kept sets: in every image the GPU keeps its own budget k of tokens; the oracle's top k
    # by its own scores must be the same set up to near-ties (a GPU-only token within the
    # score tolerance of an oracle-only one)
    got_set = set(ref["kept_idx"].tolist())
    for r in range(lay.n_requests):
        for i in range(int(lay.img_cu[r]), int(lay.img_cu[r + 1])):
            s = int(lay.cu_seqlens[r]) + int(lay.img_start[i])
            rows = list(range(s, s + int(lay.img_len[i])))
            k = int(ref["budgets"][i])
            order = sorted(rows, key=lambda t: O.rank_key(float(s_ref[t]), t))
            top = set(order[:k])
            only_gpu = [t for t in rows if t in got_set and t not in top]
            only_ref = [t for t in rows if t in top and t not in got_set]
            assert len(only_gpu) == len(only_ref), i
            for a in only_gpu:
                assert any(near_tie(float(s_ref[a]), float(s_ref[b])) for b in only_ref), (i, a)


def test_prune_fused_selection_ties_nan_and_sizes():
    # image sizes around every sort size of the fused kernel (256, 512, 1024) and past it
    # (radix path); rows with h_cur == h_prior score within a few ulps of 0 (many exact
    # ties), rows with an inf entry score NaN, duplicated rows give equal scores at
    # distant positions
    sizes = [1, 7, 255, 256, 257, 511, 512, 513, 1023, 1024, 1025, 2100]
    reqs = [[("t", 5)] + sum([[("i", n), ("t", 2)] for n in sizes[:6]], []),
            [("t", 1)] + sum([[("i", n), ("t", 1)] for n in sizes[6:]], [])]
    wl = synth.make_custom(reqs, keep_ratio=0.4, parts=("A", "pos"))
    rng = np.random.default_rng(21)
    h_cur, h_prior = wl.tensors["h_cur"].copy(), wl.tensors["h_prior"].copy()
    vis = np.flatnonzero(wl.layout.visual_mask())
    same = rng.choice(vis, size=len(vis) // 5, replace=False)
    h_cur[same] = h_prior[same]
    nan_rows = rng.choice(np.setdiff1d(vis, same), size=40, replace=False)
    h_cur[nan_rows, 3] = 0x7F80  # +inf in bf16
    free = np.setdiff1d(vis, np.concatenate([same, nan_rows]))
    dup_src = rng.choice(vis, size=200)
    dup_dst = rng.choice(free, size=200, replace=False)
    h_cur[dup_dst], h_prior[dup_dst] = h_cur[dup_src], h_prior[dup_src]
    wl.tensors["h_cur"], wl.tensors["h_prior"] = h_cur, h_prior
    dw = DevWorkload(wl)
    for kr in (0.05, 0.4, 0.95):
        krs = np.full(wl.layout.n_requests, kr, dtype=np.float32)
        out = avtp.prune(dw.L, "hidden_variation", keep_ratio=torch.from_numpy(krs).cuda(), keep_ratio_host=krs,
                         planes={"pos": dw.t["pos"]}, **dw.score_tensors("hidden_variation"))
        torch.cuda.synchronize()
        assert avtp.read_device_status(out.workspace) == avtp.OK
        got = out.scores.cpu().numpy()
        # equal rows score 1 - cos within a few fp32 ulps of 0: many exact ties
        assert np.isnan(got[nan_rows]).all() and (np.abs(got[same]) < 1e-6).all()
        ref = O.prune(wl.layout, keep_ratio=krs, scores_f32=got, planes={"pos": wl.pos})
        assert np.array_equal(out.budgets[:wl.layout.n_images].cpu().numpy(), ref["budgets"])
        assert np.array_equal(out.kept_idx.cpu().numpy(), ref["kept_idx"]), kr
        assert np.array_equal(out.outputs["pos"].cpu().numpy(), ref["pos"])


def test_prune_repeatable_and_deterministic():
    wl, dw = workload("qwen3_vl_8b")
    call = avtp.PruneCall(dw.L, "hidden_variation", keep_ratio=dw.keep_ratio, keep_ratio_host=wl.keep_ratio,
                          rows={"hidden": dw.t["h_cur"]}, planes={"pos": dw.t["pos"]},
                          **dw.score_tensors("hidden_variation"))
    first = None
    for _ in range(3):
        b = call.run()
        torch.cuda.synchronize()
        snap = (b.scores.cpu().numpy().copy(), b.img_sums.cpu().numpy().copy(), b.kept_idx.cpu().numpy().copy())
        if first is None:
            first = snap
        else:
            for x, y in zip(first, snap):
                assert np.array_equal(x, y)


# ---------------------------------------------------------------- device-side validation
def _status_after(fn):
    ws = avtp.new_workspace(1 << 20)
    fn(ws)
    torch.cuda.synchronize()
    return avtp.read_device_status(ws)


def test_device_rejects_bad_spans():
    h_cur = torch.randn(20, 64, device="cuda").to(torch.bfloat16)
    for starts, lens in [([0, 10], [12, 5]),      # overlapping spans
                         ([15], [10]),            # past the request end
                         ([3], [0])]:             # empty image
        L = avtp.Layout.from_host([0, 20], [0, len(starts)], starts, lens)
        st = _status_after(lambda ws: avtp.score(L, "hidden_variation", h_cur=h_cur, h_prior=h_cur, workspace=ws))
        assert st == avtp.ERR_DEVICE_INPUT


def test_device_rejects_bad_keep_ratio_and_budgets():
    L = avtp.Layout.from_host([0, 20], [0, 1], [2], [10])
    sums = torch.zeros(1, dtype=torch.int64, device="cuda")
    for kr in (1.5, 0.01, 0.96):  # above 1, below r_min = 0.05, above r_max = 0.95
        st = _status_after(lambda ws: avtp.allocate(L, sums, torch.tensor([kr], device="cuda"), workspace=ws))
        assert st == avtp.ERR_DEVICE_INPUT
    scores = torch.zeros(20, device="cuda")
    out_cu = torch.tensor([0, 30], dtype=torch.int32, device="cuda")
    bad_budget = torch.tensor([11], dtype=torch.int32, device="cuda")
    st = _status_after(lambda ws: avtp.select(L, scores, bad_budget, out_cu, 30, workspace=ws))
    assert st == avtp.ERR_DEVICE_INPUT


def test_device_rejects_out_of_range_kept_index():
    src = torch.randn(10, 64, device="cuda").to(torch.bfloat16)
    out = torch.zeros(3, 64, dtype=torch.bfloat16, device="cuda")
    idx = torch.tensor([1, 10, 2], dtype=torch.int32, device="cuda")
    st = _status_after(lambda ws: avtp.compact(idx, 10, [(src, out)], workspace=ws))
    assert st == avtp.ERR_DEVICE_INPUT
    assert torch.equal(out[0].cpu(), src[1].cpu()) and torch.equal(out[2].cpu(), src[2].cpu())


def test_host_rejects_bad_arguments():
    L = avtp.Layout.from_host([0, 20], [0, 1], [2], [10])
    x = torch.randn(20, 60, device="cuda").to(torch.bfloat16)  # hidden 60: not a multiple of 8
    with pytest.raises(avtp.AVTPError) as e:
        avtp.score(L, "hidden_variation", h_cur=x, h_prior=x)
    assert e.value.code == avtp.ERR_UNSUPPORTED
    q = torch.randn(20, 4, 96, device="cuda").to(torch.bfloat16)  # head_dim 96
    with pytest.raises(avtp.AVTPError) as e:
        avtp.score(L, "text_attention", q=q, k=q[:, :2].contiguous())
    assert e.value.code == avtp.ERR_UNSUPPORTED
    with pytest.raises(avtp.AVTPError) as e:
        avtp.score(L, "hidden_variation", h_cur=x[:, :56].contiguous(), h_prior=x[:, :56].contiguous(),
                   workspace=avtp.new_workspace(256))
    assert e.value.code == avtp.ERR_WORKSPACE
