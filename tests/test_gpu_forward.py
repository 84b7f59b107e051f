"""GPU parity of the layer's causal attention forward (avtp_attn_forward) and of the
text-attention scores it produces from its own LSE, against the fp64 oracle.

Tolerances, from the arithmetic:
- LSE: rel 1e-3 / abs 1e-5. The kernel sums fp32 exponentials of fp32 logits of bf16
  inputs, so its error is near fp32 rounding.
- O: |O - O_ref| <= 2^-8 * O_abs + 1e-5 element by element, where O_abs is the forward
  of |v|. The kernel rounds each probability p to bf16 before P V (as FlashAttention
  does), and bf16 rounding moves p by at most 2^-8 p, so the weighted sum moves by at
  most 2^-8 sum p |v| / l. The rounding errors are of both signs, so their mean over
  all elements must also stay below 2^-10 * O_abs.
- Scores: rel 1e-3 / abs 1e-5, as for avtp_score; image sums exact for the GPU's
  own scores.
"""
import numpy as np
import pytest
import torch

from oracle import avtp_oracle as O
from paper_2608_26806_gb300 import avtp, synth
from tests.gpu_util import ATOL, RTOL, assert_scores_close, bf16_dev, dev_layout, ensure_built

pytestmark = pytest.mark.gpu

O_REL = 2.0 ** -8
O_MEAN_REL = 2.0 ** -10


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    ensure_built()


def _dev(wl):
    L = dev_layout(wl.layout)
    return L, bf16_dev(wl.q), bf16_dev(wl.k), bf16_dev(wl.v)


def _check_o(got, ref, ref_abs):
    err = np.abs(got - ref)
    bound = O_REL * ref_abs + 1e-5
    worst = np.argmax(err - bound)
    assert np.all(err <= bound), (f"O outside its bound at {np.unravel_index(worst, err.shape)}: "
                                  f"{got.flat[worst]} vs {ref.flat[worst]} (bound {bound.flat[worst]})")
    assert err.sum() <= O_MEAN_REL * ref_abs.sum() + 1e-7 * err.size


def _abs_v(v_bits):
    return (v_bits & np.uint16(0x7FFF)).astype(np.uint16)


# Layouts for the forward: requests of 1, 127, 128, 129 and several hundred tokens that
# start at packed offsets that are not multiples of 128 (so query tiles and key blocks
# straddle request boundaries), text only, images only, and many query tiles.
_FWD_LAYOUTS = [
    [[("t", 1)]],
    [[("i", 64), ("t", 63)], [("t", 1), ("i", 127), ("t", 1)], [("i", 200), ("t", 57)], [("t", 128)]],
    [[("t", 5), ("i", 300), ("t", 3)], [("i", 128)], [("t", 130), ("i", 385), ("t", 2)]],
    [[("t", 70), ("i", 129), ("i", 1), ("t", 1)], [("i", 40), ("t", 3), ("i", 600), ("t", 100)]],
]


@pytest.mark.parametrize("layout_id", range(len(_FWD_LAYOUTS)))
@pytest.mark.parametrize("heads", [(4, 4, 64), (6, 2, 64), (12, 4, 128), (7, 1, 128)])
def test_forward_matches_oracle(layout_id, heads):
    Hq, Hkv, d = heads
    wl = synth.make_custom(_FWD_LAYOUTS[layout_id], n_q_heads=Hq, n_kv_heads=Hkv, head_dim=d, hidden=64,
                           seed=31 + layout_id, parts=("B", "V"))
    L, q, k, v = _dev(wl)
    o, lse, scores, sums = avtp.attn_forward(L, q=q, k=k, v=v, softmax_scale=wl.softmax_scale)
    torch.cuda.synchronize()
    ref_o, ref_lse = O.attention_forward(wl.layout, wl.q, wl.k, wl.v, Hq, Hkv, wl.softmax_scale)
    ref_abs, _ = O.attention_forward(wl.layout, wl.q, wl.k, _abs_v(wl.v), Hq, Hkv, wl.softmax_scale)
    _check_o(o.cpu().numpy(), ref_o, ref_abs)
    np.testing.assert_allclose(lse.cpu().numpy(), ref_lse, rtol=RTOL, atol=ATOL)
    # criterion B from the forward's LSE
    got = scores.cpu().numpy()
    vis = wl.layout.visual_mask()
    if vis.any():
        ref = O.score_text_attention(wl.layout, wl.q, wl.k, Hq, Hkv, wl.softmax_scale)
        assert_scores_close(got, ref, vis)
        assert np.array_equal(sums.cpu().numpy(), O.image_sums(wl.layout, got))


@pytest.mark.parametrize("query_set,path", [("text", "tensor"), ("text", "cuda"), ("last", "auto")])
def test_forward_side_output_on_each_scoring_path(query_set, path):
    wl = synth.make_custom(_FWD_LAYOUTS[2], n_q_heads=8, n_kv_heads=2, head_dim=128, hidden=64, seed=5,
                           parts=("B", "V"))
    L, q, k, v = _dev(wl)
    _, lse, scores, sums = avtp.attn_forward(L, q=q, k=k, v=v, softmax_scale=wl.softmax_scale, query_set=query_set,
                                             path=path)
    torch.cuda.synchronize()
    got = scores.cpu().numpy()
    ref = O.score_text_attention(wl.layout, wl.q, wl.k, 8, 2, wl.softmax_scale, query_set=query_set)
    assert_scores_close(got, ref, wl.layout.visual_mask())
    assert np.array_equal(sums.cpu().numpy(), O.image_sums(wl.layout, got))


def test_plain_forward_leaves_scores_alone():
    wl = synth.make_custom(_FWD_LAYOUTS[1], n_q_heads=4, n_kv_heads=2, head_dim=64, hidden=64, seed=9,
                           parts=("B", "V"))
    L, q, k, v = _dev(wl)
    o, lse, scores, sums = avtp.attn_forward(L, q=q, k=k, v=v, softmax_scale=wl.softmax_scale, scores=False)
    torch.cuda.synchronize()
    assert scores is None and sums is None
    ref_o, ref_lse = O.attention_forward(wl.layout, wl.q, wl.k, wl.v, 4, 2, wl.softmax_scale)
    ref_abs, _ = O.attention_forward(wl.layout, wl.q, wl.k, _abs_v(wl.v), 4, 2, wl.softmax_scale)
    _check_o(o.cpu().numpy(), ref_o, ref_abs)
    np.testing.assert_allclose(lse.cpu().numpy(), ref_lse, rtol=RTOL, atol=ATOL)


def test_forward_repeatable():
    wl = synth.make_custom(_FWD_LAYOUTS[3], n_q_heads=6, n_kv_heads=2, head_dim=128, hidden=64, seed=3,
                           parts=("B", "V"))
    L, q, k, v = _dev(wl)
    c = avtp.ForwardCall(L, q=q, k=k, v=v, softmax_scale=wl.softmax_scale)
    c.run()
    o1, l1, s1 = c.o.clone(), c.lse.clone(), c.scores.clone()
    c.run()
    torch.cuda.synchronize()
    assert torch.equal(o1, c.o) and torch.equal(l1, c.lse) and torch.equal(s1, c.scores)
    assert avtp.read_device_status(c.workspace) == 0


# ---------------------------------------------------------------- full-size workloads
@pytest.mark.parametrize("name", ["qwen3_vl_8b", "llava_ov_7b"])
def test_forward_full_size_sampled_rows(name):
    """The workload the bench times: O and the LSE of sampled rows (the first and last rows
    of query tiles, the request's last token) against the oracle's per-row forward, the
    LSE of every text query against the oracle's, and the scores in full."""
    wl = synth.make_workload(name, parts=("B", "V"))
    L, q, k, v = _dev(wl)
    Hq, Hkv = wl.n_q_heads, wl.n_kv_heads
    o, lse, scores, sums = avtp.attn_forward(L, q=q, k=k, v=v, softmax_scale=wl.softmax_scale)
    torch.cuda.synchronize()
    T = wl.layout.n_tokens
    rows = sorted({0, 1, 127, 128, 129, 2047, 2048, T // 2, T - 129, T - 128, T - 2, T - 1})
    ref_o, ref_lse = O.attention_forward_rows(wl.layout, wl.q, wl.k, wl.v, Hq, Hkv, wl.softmax_scale, 0, rows)
    ref_abs, _ = O.attention_forward_rows(wl.layout, wl.q, wl.k, _abs_v(wl.v), Hq, Hkv, wl.softmax_scale, 0, rows)
    _check_o(o[rows].cpu().numpy(), ref_o, ref_abs)
    np.testing.assert_allclose(lse[:, rows].cpu().numpy(), ref_lse, rtol=RTOL, atol=ATOL)
    text = ~wl.layout.visual_mask()
    ref_text_lse = O.text_lse(wl.layout, wl.q, wl.k, Hq, Hkv, wl.softmax_scale)
    np.testing.assert_allclose(lse.cpu().numpy()[:, text], ref_text_lse[:, text], rtol=RTOL, atol=ATOL)
    got = scores.cpu().numpy()
    ref = O.score_text_attention(wl.layout, wl.q, wl.k, Hq, Hkv, wl.softmax_scale)
    assert_scores_close(got, ref, wl.layout.visual_mask())
    assert np.array_equal(sums.cpu().numpy(), O.image_sums(wl.layout, got))


def test_forward_serving_batch_sampled_rows():
    """Eight varlen requests: sampled rows of every request (its first, tile-edge and last
    tokens) against the oracle."""
    wl = synth.make_workload("internvl3_5_8b", parts=("B", "V"))
    L, q, k, v = _dev(wl)
    Hq, Hkv = wl.n_q_heads, wl.n_kv_heads
    o, lse, _, _ = avtp.attn_forward(L, q=q, k=k, v=v, softmax_scale=wl.softmax_scale, scores=False)
    torch.cuda.synchronize()
    cu = wl.layout.cu_seqlens
    o_h, lse_h = o.cpu().numpy(), lse.cpu().numpy()
    for r in range(wl.layout.n_requests):
        n = int(cu[r + 1] - cu[r])
        rows = sorted({0, 127, 128, n // 2, n - 1})
        ref_o, ref_lse = O.attention_forward_rows(wl.layout, wl.q, wl.k, wl.v, Hq, Hkv, wl.softmax_scale, r, rows)
        ref_abs, _ = O.attention_forward_rows(wl.layout, wl.q, wl.k, _abs_v(wl.v), Hq, Hkv, wl.softmax_scale, r,
                                              rows)
        g = [int(cu[r]) + p for p in rows]
        _check_o(o_h[g], ref_o, ref_abs)
        np.testing.assert_allclose(lse_h[:, g], ref_lse, rtol=RTOL, atol=ATOL)


def test_forward_many_small_requests():
    """Forty requests of 1 to 300 tokens: many query tiles per call, tiles and key blocks
    that straddle request boundaries at every offset, requests shorter than a tile."""
    rng = np.random.default_rng(17)
    reqs = []
    for _ in range(40):
        segs = []
        for _ in range(int(rng.integers(1, 4))):
            segs.append(("t" if rng.random() < 0.5 else "i", int(rng.integers(1, 101))))
        reqs.append(segs)
    wl = synth.make_custom(reqs, n_q_heads=4, n_kv_heads=1, head_dim=64, hidden=64, seed=23, parts=("B", "V"))
    L, q, k, v = _dev(wl)
    o, lse, scores, sums = avtp.attn_forward(L, q=q, k=k, v=v, softmax_scale=wl.softmax_scale)
    torch.cuda.synchronize()
    ref_o, ref_lse = O.attention_forward(wl.layout, wl.q, wl.k, wl.v, 4, 1, wl.softmax_scale)
    ref_abs, _ = O.attention_forward(wl.layout, wl.q, wl.k, _abs_v(wl.v), 4, 1, wl.softmax_scale)
    _check_o(o.cpu().numpy(), ref_o, ref_abs)
    np.testing.assert_allclose(lse.cpu().numpy(), ref_lse, rtol=RTOL, atol=ATOL)
    vis = wl.layout.visual_mask()
    ref = O.score_text_attention(wl.layout, wl.q, wl.k, 4, 1, wl.softmax_scale)
    assert_scores_close(scores.cpu().numpy(), ref, vis)


def test_forward_strided_tensors():
    """q, k and v rows with padded token strides, O and the LSE written into wider buffers:
    the strides of the ABI are honoured and nothing outside the views is written."""
    Hq, Hkv, d = 6, 2, 128
    wl = synth.make_custom(_FWD_LAYOUTS[2], n_q_heads=Hq, n_kv_heads=Hkv, head_dim=d, hidden=64, seed=41,
                           parts=("B", "V"))
    T = wl.layout.n_tokens
    L = dev_layout(wl.layout)

    def padded(bits, heads):
        big = torch.zeros(T, heads + 1, d, dtype=torch.bfloat16, device="cuda")
        big[:, :heads] = bf16_dev(bits)
        return big[:, :heads]

    q, k, v = padded(wl.q, Hq), padded(wl.k, Hkv), padded(wl.v, Hkv)
    o_big = torch.full((T, Hq + 2, d), 7.0, dtype=torch.float32, device="cuda")
    lse_big = torch.full((Hq, T + 24), 7.0, dtype=torch.float32, device="cuda")
    c = avtp.ForwardCall(L, q=q, k=k, v=v, softmax_scale=wl.softmax_scale, o=o_big[:, :Hq], lse=lse_big[:, :T])
    c.run()
    torch.cuda.synchronize()
    ref_o, ref_lse = O.attention_forward(wl.layout, wl.q, wl.k, wl.v, Hq, Hkv, wl.softmax_scale)
    ref_abs, _ = O.attention_forward(wl.layout, wl.q, wl.k, _abs_v(wl.v), Hq, Hkv, wl.softmax_scale)
    _check_o(o_big[:, :Hq].cpu().numpy(), ref_o, ref_abs)
    np.testing.assert_allclose(lse_big[:, :T].cpu().numpy(), ref_lse, rtol=RTOL, atol=ATOL)
    assert torch.all(o_big[:, Hq:] == 7.0) and torch.all(lse_big[:, T:] == 7.0)
    ref = O.score_text_attention(wl.layout, wl.q, wl.k, Hq, Hkv, wl.softmax_scale)
    assert_scores_close(c.scores.cpu().numpy(), ref, wl.layout.visual_mask())
