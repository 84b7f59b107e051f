"""GPU parity on the long multi-image stress workload, at full size.

4 requests x 64 images x 1024 visual tokens (+512 text tokens each), hidden 4096,
32/8 heads of 128: 264,192 tokens, about 8 GB on the device. The requests are
independent, so the oracle scores them one at a time: criterion A on every visual row
of all four requests, criterion B on every visual key of requests 0 and 3 (the full
causal attention of each). Request 3's rows of h_cur start past 2^31 bytes and its text
queries too, where a 32-bit offset would show. Steps 2-4 are checked on the whole batch
fed the GPU's own scores: budgets, kept indices and the gathered rows bit-exact.
"""
import numpy as np
import pytest
import torch

from oracle import avtp_oracle as O
from paper_2608_26806_gb300 import avtp, synth
from tests.gpu_util import ATOL, RTOL, DevWorkload, bits_of, ensure_built

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def long_workload():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    ensure_built()
    wl = synth.make_workload("long")
    dw = DevWorkload(wl)
    yield wl, dw
    del dw
    torch.cuda.empty_cache()


def _request(wl, r):
    """Layout of request r alone and its packed token range [a, b)."""
    lay = wl.layout
    a, b = int(lay.cu_seqlens[r]), int(lay.cu_seqlens[r + 1])
    i0, i1 = int(lay.img_cu[r]), int(lay.img_cu[r + 1])
    sub = synth.Layout(cu_seqlens=np.array([0, b - a], dtype=np.int32), img_cu=np.array([0, i1 - i0], dtype=np.int32),
                       img_start=lay.img_start[i0:i1].copy(), img_len=lay.img_len[i0:i1].copy())
    return sub, a, b


def test_score_long_workload_last_token(long_workload):
    # the last-token query set on the CUDA-core path: every visual key of all four requests
    wl, dw = long_workload
    lay = wl.layout
    scores, sums = avtp.score(dw.L, "text_attention", query_set="last", **dw.score_tensors("text_attention"))
    torch.cuda.synchronize()
    got = scores.cpu().numpy()
    ref = O.score_text_attention(lay, wl.q, wl.k, wl.n_q_heads, wl.n_kv_heads, wl.softmax_scale, query_set="last")
    vis = lay.visual_mask()
    np.testing.assert_allclose(got[vis], ref[vis], rtol=RTOL, atol=ATOL)
    assert np.array_equal(sums.cpu().numpy(), O.image_sums(lay, got))


@pytest.mark.parametrize("criterion", ["hidden_variation", "text_attention"])
def test_prune_long_workload(long_workload, criterion):
    wl, dw = long_workload
    lay = wl.layout
    relative = criterion == "text_attention"
    out = avtp.prune(dw.L, criterion, keep_ratio=dw.keep_ratio, keep_ratio_host=wl.keep_ratio,
                     rows={"hidden": dw.t["h_cur"]}, planes={"pos": dw.t["pos"]}, **dw.score_tensors(criterion))
    torch.cuda.synchronize()
    assert avtp.read_device_status(out.workspace) == avtp.OK
    got = out.scores.cpu().numpy()

    # step 1 against the oracle, request by request
    row_bytes = wl.h_cur.shape[1] * 2
    requests = range(lay.n_requests) if criterion == "hidden_variation" else (0, lay.n_requests - 1)
    for r in requests:
        sub, a, b = _request(wl, r)
        if r == lay.n_requests - 1:
            assert b * row_bytes > 2 ** 31  # the last request's rows end past 2^31 bytes
        if criterion == "hidden_variation":
            ref = O.score_hidden_variation(sub, wl.h_cur[a:b], wl.h_prior[a:b])
        else:
            ref = O.score_text_attention(sub, wl.q[a:b], wl.k[a:b], wl.n_q_heads, wl.n_kv_heads, wl.softmax_scale)
        vis = sub.visual_mask()
        np.testing.assert_allclose(got[a:b][vis], ref[vis], rtol=RTOL, atol=ATOL, err_msg=f"request {r}")

    # steps 2-4 on the whole batch, fed the GPU's scores: bit-exact
    exp = O.prune(lay, keep_ratio=wl.keep_ratio, scores_f32=got, relative=relative, planes={"pos": wl.pos})
    assert np.array_equal(out.img_sums[:lay.n_images].cpu().numpy(), exp["img_sums"])
    assert np.array_equal(out.budgets[:lay.n_images].cpu().numpy(), exp["budgets"])
    assert np.array_equal(out.out_cu_seqlens.cpu().numpy(), exp["out_cu_seqlens"])
    kept = out.kept_idx.cpu().numpy()
    assert np.array_equal(kept, exp["kept_idx"])
    assert np.array_equal(out.outputs["pos"].cpu().numpy(), exp["pos"])
    # the gathered hidden rows: every row, compared as bit patterns
    hid = bits_of(out.outputs["hidden"])
    assert np.array_equal(hid, wl.h_cur[kept.astype(np.int64)])
    # the two strong images of each request keep more than the weak ones
    if criterion == "hidden_variation":
        b = exp["budgets"].reshape(lay.n_requests, -1)
        strong = wl.signal.reshape(lay.n_requests, -1) > 1.0
        assert np.all(b[strong].min() > b[~strong].max())


def test_attention_forward_long_workload(long_workload):
    """The layer's attention forward over all 264,192 tokens: sampled rows (tile edges, the
    middle, the last token) of requests 0 and 3 against the oracle's per-row forward, at
    the bound of the bf16 probabilities (2^-8 of the forward of |v|). Request 3's rows of O
    start 3.2 GB into the output, past 2^31 bytes, where a 32-bit offset would show. Criterion B's scores from the
    forward's LSE on every visual key of request 3."""
    wl, dw = long_workload
    lay = wl.layout
    synth.build_tensors(wl, parts=("V",))  # the values only; the other tensors stay as drawn
    v = torch.from_numpy(np.ascontiguousarray(wl.v).view(np.int16)).cuda().view(torch.bfloat16)
    Hq, Hkv = wl.n_q_heads, wl.n_kv_heads
    o, lse, scores, _ = avtp.attn_forward(dw.L, q=dw.t["q"], k=dw.t["k"], v=v, softmax_scale=wl.softmax_scale)
    torch.cuda.synchronize()
    v_abs = (wl.v & np.uint16(0x7FFF)).astype(np.uint16)
    for r in (0, lay.n_requests - 1):
        a, b = int(lay.cu_seqlens[r]), int(lay.cu_seqlens[r + 1])
        n = b - a
        if r == lay.n_requests - 1:
            assert a * Hq * wl.head_dim * 4 > 2 ** 31  # O rows of the last request start past 2^31 bytes
        rows = sorted({0, 127, 128, n // 2, n - 129, n - 1})
        ref_o, ref_lse = O.attention_forward_rows(lay, wl.q, wl.k, wl.v, Hq, Hkv, wl.softmax_scale, r, rows)
        ref_abs, _ = O.attention_forward_rows(lay, wl.q, wl.k, v_abs, Hq, Hkv, wl.softmax_scale, r, rows)
        g = [a + p for p in rows]
        got_o = o[g].cpu().numpy()
        assert np.all(np.abs(got_o - ref_o) <= 2.0 ** -8 * ref_abs + 1e-5), f"request {r}"
        np.testing.assert_allclose(lse[:, g].cpu().numpy(), ref_lse, rtol=RTOL, atol=ATOL, err_msg=f"request {r}")
    sub, a, b = _request(wl, lay.n_requests - 1)
    ref = O.score_text_attention(sub, wl.q[a:b], wl.k[a:b], Hq, Hkv, wl.softmax_scale)
    vis = sub.visual_mask()
    np.testing.assert_allclose(scores.cpu().numpy()[a:b][vis], ref[vis], rtol=RTOL, atol=ATOL)
    del o, lse, scores, v
    wl.tensors.pop("v")
    torch.cuda.empty_cache()
