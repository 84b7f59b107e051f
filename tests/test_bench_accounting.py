"""The bench's algorithmic bytes and FLOPs (the numerators of its rooflines), checked on
the CPU against a hand count and against brute-force counts over explicit causal masks."""
import os
import sys
from types import SimpleNamespace

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2608_26806_gb300 import synth  # noqa: E402


def _wl(segs, D=8, Hq=2, Hkv=1, d=4, P=1):
    return SimpleNamespace(layout=synth.Layout.from_segments(segs), hidden=D, pos_planes=P, n_q_heads=Hq,
                           n_kv_heads=Hkv, head_dim=d)


def test_hand_counted_example():
    # text at request-local positions 0, 1 and 5; visual tokens at 2..4
    wl = _wl([[("t", 2), ("i", 3), ("t", 1)]])
    n_kept = 4  # three text tokens and one visual token
    a = bench.stage_accounting(wl, "hidden_variation", n_kept)
    assert a["n_vis"] == 3 and a["n_txt"] == 3
    assert a["score_bytes"] == 2 * 3 * 8 * 2
    assert a["stage_bytes"] == 96 + 3 * 8 * 2 + 4 * 8 * 2 + 4 * 4 * 2
    assert a["flops"] == 0
    # pass 1: the text queries see 1, 2 and 6 keys; pass 2: 0, 0 and 3 visual keys
    b = bench.stage_accounting(wl, "text_attention", n_kept)
    assert b["flops"] == 2 * 2 * 4 * (1 + 2 + 6) + 2 * 2 * 4 * (0 + 0 + 3)
    assert b["score_bytes"] == 6 * 1 * 4 * 2 + 3 * 2 * 4 * 2
    bl = bench.stage_accounting(wl, "text_attention", n_kept, lse=True)
    assert bl["flops"] == 2 * 2 * 4 * 3
    assert bl["score_bytes"] == 3 * 1 * 4 * 2 + 3 * 2 * 4 * 2 + 3 * 2 * 4


def test_last_token_accounting_by_hand():
    # the request's last token as the only query: every key once, one query row per head;
    # FMAs (not tensor-core FLOPs): the 6 keys it sees in pass 1, the 3 visual keys in pass 2
    wl = _wl([[("t", 2), ("i", 3), ("t", 1)]])
    c = bench.stage_accounting(wl, "text_attention", 4, query_set="last")
    assert c["score_bytes"] == 6 * 1 * 4 * 2 + 1 * 2 * 4 * 2
    assert c["stage_bytes"] == c["score_bytes"] + 3 * 8 * 2 + 4 * 8 * 2 + 4 * 4 * 2
    assert c["flops"] == 0
    assert c["fma_flops"] == 2 * 2 * 4 * 6 + 2 * 2 * 4 * 3


def test_flops_equal_brute_force_mask_counts():
    rng = np.random.default_rng(4)
    for _ in range(40):
        reqs = []
        for _ in range(int(rng.integers(1, 4))):
            segs = [("i" if rng.random() < 0.5 else "t", int(rng.integers(1, 7))) for _ in range(int(rng.integers(1, 6)))]
            reqs.append(segs)
        Hq, d = int(rng.choice([2, 4, 8])), int(rng.choice([4, 8]))
        wl = _wl(reqs, Hq=Hq, Hkv=1, d=d)
        lay = wl.layout
        vis = lay.visual_mask()
        p1 = p2 = 0
        for r in range(lay.n_requests):
            a, b = int(lay.cu_seqlens[r]), int(lay.cu_seqlens[r + 1])
            n = b - a
            causal = np.tril(np.ones((n, n), dtype=bool))  # [query, key]: key <= query
            text_q = ~vis[a:b]
            p1 += int(causal[text_q].sum())
            p2 += int(causal[text_q][:, vis[a:b]].sum())
        got = bench.stage_accounting(wl, "text_attention", 0)["flops"]
        assert got == 2 * Hq * d * (p1 + p2)
        got_lse = bench.stage_accounting(wl, "text_attention", 0, lse=True)["flops"]
        assert got_lse == 2 * Hq * d * p2


def test_stage_roofline_takes_the_slower_bound():
    # 6794.1 kB at 6794.1 GB/s is 1 us; 1.91 MFLOP at 1910 TFLOP/s is 1 ns
    acct = {"stage_bytes": 6_794_100, "flops": 1_910_000}
    r = bench.stage_roofline(acct, 0.002, 6794.1, 1910.0, "measured")
    assert r["bound"] == "hbm"
    assert abs(r["bound_us"] - 1.0) < 1e-9
    assert abs(r["frac"] - 0.5) < 1e-4
    acct = {"stage_bytes": 6_794, "flops": 1_910_000_000}  # 1 ns of bytes, 1 us of FLOPs
    r = bench.stage_roofline(acct, 0.004, 6794.1, 1910.0, "measured")
    assert r["bound"] == "tensor"
    assert abs(r["frac"] - 0.25) < 1e-4


def test_forward_flops_equal_brute_force_mask_counts():
    # the forward's FLOPs: Q K^T and P V, 2 d each per query head and visible (query, key)
    # pair, pairs counted from an explicit causal mask per request
    rng = np.random.default_rng(5)
    for _ in range(20):
        reqs = [[("t", int(rng.integers(1, 9))), ("i", int(rng.integers(1, 9)))] for _ in range(int(rng.integers(1, 4)))]
        wl = _wl(reqs, Hq=int(rng.integers(1, 5)), d=int(rng.choice([4, 8])))
        cu = wl.layout.cu_seqlens
        pairs = 0
        for r in range(len(cu) - 1):
            n = int(cu[r + 1] - cu[r])
            pairs += int(np.tril(np.ones((n, n), dtype=np.int64)).sum())
        assert bench.forward_flops(wl) == 4 * wl.head_dim * wl.n_q_heads * pairs
    # the Qwen3-VL-8B-shaped request: 796 GFLOP
    q3 = synth.make_workload("qwen3_vl_8b", parts=())
    assert bench.forward_flops(q3) == 795_857_649_664
