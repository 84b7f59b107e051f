"""GPU parity of progressive pruning: the stage run three times on a shrinking batch.

Paper §3.3.2 prunes at several layers in a progressive schedule; at each pruning point
the hidden states of the previous one, compacted to the surviving tokens, are h_prior
(§3.3.1). The next stage's layout is built on the device by avtp_pruned_layout. Each
stage is checked against the oracle chained the same way: the layout exactly, scores to
rel 1e-3 / abs 1e-5, and budgets, kept indices and compacted rows bit-exact when both
sides are fed the GPU's scores. The per-stage keep ratio is 0.5^(1/3), so that half of
the visual tokens survive the three stages (the paper keeps 50 % overall and does not
give a per-layer schedule).
"""
import numpy as np
import pytest
import torch

from oracle import avtp_oracle as O
from paper_2608_26806_gb300 import avtp, synth
from tests.gpu_util import assert_scores_close, bf16_dev, bits_of, ensure_built

pytestmark = pytest.mark.gpu

STAGES = 3
STAGE_RATIO = np.float32(0.5 ** (1.0 / 3.0))


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    ensure_built()


def _next_hidden(h_prior_bits: np.ndarray, seed: int) -> np.ndarray:
    """The next pruning layer's hidden states: h_prior + 0.5 * N(0,1), rounded to bf16."""
    rng = np.random.default_rng(seed)
    z = rng.standard_normal(h_prior_bits.shape).astype(np.float32)
    return synth.f32_to_bf16_bits(synth.bf16_bits_to_f32(h_prior_bits) + 0.5 * z)


@pytest.mark.parametrize("name", ["tiny", "qwen3_vl_8b"])
def test_progressive_pruning_three_stages(name):
    wl = synth.make_workload(name, parts=("A", "pos"))
    lay_host = wl.layout
    L = avtp.Layout.from_host(lay_host.cu_seqlens, lay_host.img_cu, lay_host.img_start, lay_host.img_len)
    h_cur, h_prior, pos = wl.h_cur, wl.h_prior, wl.pos
    ratio = np.full(lay_host.n_requests, STAGE_RATIO, dtype=np.float32)
    for stage in range(STAGES):
        kr = torch.from_numpy(ratio).cuda()
        out = avtp.prune(L, "hidden_variation", keep_ratio=kr, keep_ratio_host=ratio, h_cur=bf16_dev(h_cur),
                         h_prior=bf16_dev(h_prior), rows={"hidden": bf16_dev(h_cur)},
                         planes={"pos": torch.from_numpy(pos).cuda()})
        torch.cuda.synchronize()
        assert avtp.read_device_status(out.workspace) == avtp.OK
        got_scores = out.scores.cpu().numpy()
        vis = lay_host.visual_mask()
        assert_scores_close(got_scores, O.score_hidden_variation(lay_host, h_cur, h_prior), vis)
        ref = O.prune(lay_host, keep_ratio=ratio, scores_f32=got_scores, rows={"hidden": h_cur},
                      planes={"pos": pos})
        assert np.array_equal(out.budgets[:lay_host.n_images].cpu().numpy(), ref["budgets"])
        assert np.array_equal(out.out_cu_seqlens.cpu().numpy(), ref["out_cu_seqlens"])
        assert np.array_equal(out.kept_idx[:out.n_kept].cpu().numpy(), ref["kept_idx"])
        assert np.array_equal(bits_of(out.outputs["hidden"]), ref["hidden"])
        assert np.array_equal(out.outputs["pos"].cpu().numpy(), ref["pos"])
        # the pruned batch's layout, built on the device, against the one read off the kept tokens
        L2 = avtp.pruned_layout(L, ratio, out.budgets, out.out_cu_seqlens)
        torch.cuda.synchronize()
        ref_lay = O.pruned_layout(lay_host, ref["kept_idx"], ref["out_cu_seqlens"])
        assert np.array_equal(L2.img_start.cpu().numpy(), ref_lay["img_start"])
        assert np.array_equal(L2.img_len.cpu().numpy(), ref_lay["img_len"])
        assert np.array_equal(L2.host["cu_seqlens"], ref_lay["cu_seqlens"])
        assert L2.n_tokens == out.n_kept
        # next pruning point: this stage's compacted h_cur is its h_prior
        lay_host = synth.Layout(**ref_lay)
        L = L2
        h_prior = ref["hidden"]
        h_cur = _next_hidden(h_prior, seed=100 + stage)
        pos = ref["pos"]
    # three stages at 0.5^(1/3) leave about half the visual tokens of every request
    n_vis0 = wl.layout.n_visual_per_request()
    n_vis3 = lay_host.n_visual_per_request()
    assert np.all(np.abs(n_vis3 - 0.5 * n_vis0) <= 2)


def test_pruned_layout_rejects_a_budget_outside_the_image():
    L = avtp.Layout.from_host([0, 20], [0, 2], [2, 10], [5, 6])
    budgets = torch.tensor([3, 7], dtype=torch.int32, device="cuda")  # 7 > 6
    out_cu = torch.tensor([0, 19], dtype=torch.int32, device="cuda")
    ws = avtp.new_workspace(avtp.workspace_size(L))
    L2 = avtp.pruned_layout(L, np.array([0.9], dtype=np.float32), budgets, out_cu, workspace=ws)
    torch.cuda.synchronize()
    assert avtp.read_device_status(ws) == avtp.ERR_DEVICE_INPUT
    assert L2.img_start.cpu().tolist() == [2, 0] and L2.img_len.cpu().tolist() == [3, 0]
