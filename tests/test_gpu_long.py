"""GPU parity on the long multi-image stress workload, at full size.

4 requests x 64 images x 1024 visual tokens (+512 text tokens each), hidden 4096,
32/8 heads of 128: 264,192 tokens, about 8 GB on the device. The requests are
independent and identically shaped, so the oracle scores request 0 (criterion A:
every visual row; criterion B: every visual key, from the full causal attention of
that request) and checks steps 2-4 on the whole batch fed the GPU's own scores:
budgets, kept indices and the gathered rows bit-exact.
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


def _request0(wl):
    """Layout and tensors of request 0 alone (its tokens are the first T_0 packed rows)."""
    lay = wl.layout
    T0 = int(lay.cu_seqlens[1])
    n0 = int(lay.img_cu[1])
    sub = synth.Layout(cu_seqlens=np.array([0, T0], dtype=np.int32), img_cu=np.array([0, n0], dtype=np.int32),
                       img_start=lay.img_start[:n0].copy(), img_len=lay.img_len[:n0].copy())
    return sub, T0


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

    # step 1 on request 0 against the oracle
    sub, T0 = _request0(wl)
    if criterion == "hidden_variation":
        ref = O.score_hidden_variation(sub, wl.h_cur[:T0], wl.h_prior[:T0])
    else:
        ref = O.score_text_attention(sub, wl.q[:T0], wl.k[:T0], wl.n_q_heads, wl.n_kv_heads, wl.softmax_scale)
    vis0 = sub.visual_mask()
    np.testing.assert_allclose(got[:T0][vis0], ref[vis0], rtol=RTOL, atol=ATOL)

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
