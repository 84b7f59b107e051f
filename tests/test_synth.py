"""The seeded input generator against its recipe: bf16 rounding, the token layouts and
sizes of the five workloads, the per-criterion signal, and determinism. CPU only."""
import numpy as np
import pytest

from paper_2608_26806_gb300 import synth


def test_bf16_rounding_is_nearest_even_by_the_bit_recipe():
    rng = np.random.default_rng(0)
    scale = (10.0 ** rng.integers(-8, 8, 20000)).astype(np.float32)
    x = np.concatenate([rng.standard_normal(20000).astype(np.float32) * scale,
                        np.array([0.0, -0.0, 1.0, -1.0, 3.0e38, -3.0e38, 1e-40], dtype=np.float32)]).astype(np.float32)
    # exact ties: the low 16 bits are 0x8000, with even and odd upper halves
    ties = (np.arange(1000, dtype=np.uint32) << 16 | 0x8000).astype(np.uint32) + np.uint32(0x3F800000)
    x = np.concatenate([x, ties.view(np.float32)]).astype(np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    expect = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16).astype(np.uint16)
    assert np.array_equal(synth.f32_to_bf16_bits(x), expect)
    back = synth.bf16_bits_to_f32(expect)
    assert np.array_equal(back.view(np.uint32) & 0xFFFF, np.zeros_like(back.view(np.uint32)))


def _layout(name):
    return synth.make_workload(name, parts=())


def test_workload_layouts_follow_the_recipe():
    wl = _layout("tiny")
    lay = wl.layout
    assert (lay.n_tokens, lay.n_images, int(lay.n_visual_per_request().sum())) == (224, 3, 192)
    assert (wl.hidden, wl.n_q_heads, wl.n_kv_heads, wl.head_dim, wl.pos_planes) == (256, 4, 2, 64, 1)

    wl = _layout("llava_ov_7b")
    lay = wl.layout
    assert (lay.n_tokens, lay.n_images) == (8 * (8 + 729) + 64, 8)
    assert list(lay.img_start) == [8 + j * 737 for j in range(8)] and set(lay.img_len) == {729}
    assert (wl.hidden, wl.n_q_heads, wl.n_kv_heads, wl.head_dim) == (3584, 28, 4, 128)
    assert float(wl.keep_ratio[0]) == pytest.approx(0.25)

    wl = _layout("qwen3_vl_8b")
    lay = wl.layout
    n = lay.img_len
    assert lay.n_images == 16 and all(256 <= v <= 1024 and v % 64 == 0 for v in n)
    assert lay.n_tokens - int(n.sum()) == 64 + 2 * 16 + 160
    starts = 64 + 1 + np.concatenate([[0], np.cumsum(n[:-1] + 2)])
    assert np.array_equal(lay.img_start, starts)
    assert (wl.hidden, wl.n_q_heads, wl.n_kv_heads, wl.head_dim, wl.pos_planes) == (4096, 32, 8, 128, 3)
    assert float(wl.keep_ratio[0]) == pytest.approx(0.33)
    assert wl.signal.max() == pytest.approx(1.0) and wl.signal.min() > 0

    wl = _layout("internvl3_5_8b")
    lay = wl.layout
    assert lay.n_requests == 8 and set(lay.img_len) == {256}
    m = np.diff(lay.img_cu)
    t = np.diff(lay.cu_seqlens) - 256 * m
    assert m.min() >= 4 and m.max() <= 32 and t.min() >= 64 and t.max() <= 512
    assert all(np.isclose(kr, [0.25, 0.33, 0.5]).any() for kr in wl.keep_ratio.astype(np.float64))

    wl = _layout("long")
    lay = wl.layout
    assert (lay.n_requests, lay.n_images) == (4, 256) and set(lay.img_len) == {1024}
    assert lay.n_tokens == 4 * (64 * 1026 + 384)
    assert sorted(np.unique(wl.signal)) == pytest.approx([0.1, 2.0])
    assert all(int((wl.signal[r * 64:(r + 1) * 64] == np.float32(2.0)).sum()) == 2 for r in range(4))


def test_generation_is_deterministic_and_seeded():
    a = synth.make_workload("tiny")
    b = synth.make_workload("tiny")
    for name in ("h_cur", "h_prior", "q", "k", "pos"):
        assert np.array_equal(a.tensors[name], b.tensors[name])
    c = synth.make_workload("tiny", seed=12345)
    assert not np.array_equal(a.tensors["h_prior"], c.tensors["h_prior"])


def test_criterion_signals_and_position_ids():
    wl = synth.make_workload("tiny")
    lay = wl.layout
    hc = synth.bf16_bits_to_f32(wl.tensors["h_cur"]).astype(np.float64)
    hp = synth.bf16_bits_to_f32(wl.tensors["h_prior"]).astype(np.float64)
    diff = hc - hp
    vis = lay.visual_mask()
    # h_cur = h_prior + beta Z: beta 0.25 on text, 0.25 + signal_i on image i (bf16 rounding aside)
    assert np.std(diff[~vis]) == pytest.approx(0.25, rel=0.05)
    for i in range(lay.n_images):
        s = int(lay.img_start[i])
        rows = diff[s:s + int(lay.img_len[i])]
        assert np.std(rows) == pytest.approx(0.25 + float(wl.signal[i]), rel=0.05)
    T = lay.n_tokens
    pos = wl.tensors["pos"]
    assert pos.shape == (1, T) and np.array_equal(pos[0], np.arange(T))
    q = synth.bf16_bits_to_f32(wl.tensors["q"]).astype(np.float64)
    assert abs(q.mean()) < 0.05 and np.std(q) == pytest.approx(1.0, rel=0.05)
