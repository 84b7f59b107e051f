"""GPU parity of the pruning-layer selection (paper §3.3.2), through the C ABI.

Per layer, every sample's attention to its visual tokens is the sum of its fixed-point
text-attention image sums (avtp_layer_attention); the layers are then ranked per sample
and by average rank (avtp_layer_select). Both are integer arithmetic, so they are
compared bit for bit with the oracle fed the same integers; the attention sums are also
compared with the oracle's own scores within the score tolerance. The layers are
synthetic: each has its own queries and keys, with a layer-specific shift of the visual
keys toward the text queries, so that layers differ in visual attention.
"""
import numpy as np
import pytest
import torch

from oracle import avtp_oracle as O
from paper_2608_26806_gb300 import avtp, synth
from tests.gpu_util import ATOL, RTOL, DevWorkload, dev_layout, ensure_built

pytestmark = pytest.mark.gpu

SAMPLES = [[("t", 9), ("i", 70), ("t", 3), ("i", 40), ("t", 6)], [("i", 33), ("t", 12)],
           [("t", 4), ("i", 128), ("i", 17), ("t", 20)], [("t", 30), ("i", 200), ("t", 1)]]
LAYER_SHIFTS = [0.0, 2.0, 0.5, 4.0, 1.0, 8.0, 0.25]


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    ensure_built()


def test_layer_select_matches_the_oracle():
    rng = np.random.default_rng(51)
    for trial in range(30):
        N = int(rng.integers(1, 9))
        L = int(rng.choice([1, 2, 5, 36, 64, 200, avtp_max_layers()]))
        if trial % 3 == 0:
            A = rng.integers(-3, 4, size=(N, L)).astype(np.int64) * (1 << 40)  # many ties
        else:
            A = rng.integers(-2 ** 62, 2 ** 62, size=(N, L), dtype=np.int64)
        k = int(rng.integers(1, L + 1))
        rank_sum, top = avtp.layer_select(torch.from_numpy(A).cuda(), k)
        torch.cuda.synchronize()
        ref_sum, _ = O.mean_ranks(A)
        assert rank_sum.cpu().numpy().tolist() == ref_sum.tolist(), trial
        assert top.cpu().numpy().tolist() == O.select_layers(A, k).tolist(), trial


def avtp_max_layers():
    return 1024


def test_layer_select_rejects_bad_arguments():
    A = torch.zeros((2, 3), dtype=torch.int64, device="cuda")
    for k in (0, 4):
        with pytest.raises(avtp.AVTPError) as e:
            avtp.layer_select(A, k)
        assert e.value.code == avtp.ERR_INVALID_ARG
    with pytest.raises(avtp.AVTPError) as e:
        avtp.layer_select(torch.zeros((1, 1025), dtype=torch.int64, device="cuda"), 1)
    assert e.value.code == avtp.ERR_RANGE


def test_layer_statistic_end_to_end():
    lay = synth.Layout.from_segments(SAMPLES)
    L_dev = dev_layout(lay)
    n_layers = len(LAYER_SHIFTS)
    A = torch.zeros((lay.n_requests, n_layers), dtype=torch.int64, device="cuda")
    A_from_gpu_scores = np.zeros((lay.n_requests, n_layers), dtype=np.int64)
    A_oracle = np.zeros((lay.n_requests, n_layers), dtype=np.int64)
    tol = np.zeros((lay.n_requests, n_layers))
    vis = lay.visual_mask()
    for layer, shift in enumerate(LAYER_SHIFTS):
        wl = synth.make_custom(SAMPLES, n_q_heads=4, n_kv_heads=2, head_dim=64, seed=100 + layer,
                               signal=np.full(lay.n_images, shift, dtype=np.float32), parts=("B",))
        dw = DevWorkload(wl)
        scores, sums = avtp.score(dw.L, "text_attention", **dw.score_tensors("text_attention"))
        avtp.layer_attention(L_dev, sums, A, layer)
        torch.cuda.synchronize()
        got = scores.cpu().numpy()
        A_from_gpu_scores[:, layer] = O.layer_attention(lay, O.image_sums(lay, got))
        ref = O.to_fp32(O.score_text_attention(lay, wl.q, wl.k, 4, 2, wl.softmax_scale))
        A_oracle[:, layer] = O.layer_attention(lay, O.image_sums(lay, ref))
        per_tok = (ATOL + RTOL * np.abs(ref.astype(np.float64))) * 2.0 ** 32 + 1.0
        for r in range(lay.n_requests):
            a, b = int(lay.cu_seqlens[r]), int(lay.cu_seqlens[r + 1])
            tol[r, layer] = per_tok[a:b][vis[a:b]].sum()
    A_dev = A.cpu().numpy()
    # the device sums are exactly the sums of the device's own scores ...
    assert np.array_equal(A_dev, A_from_gpu_scores)
    # ... and within the score tolerance of the oracle's
    assert np.all(np.abs(A_dev - A_oracle) <= tol)
    # the ranking, bit-exact on the device's A
    k = 3
    rank_sum, top = avtp.layer_select(A, k)
    torch.cuda.synchronize()
    ref_sum, _ = O.mean_ranks(A_dev)
    assert rank_sum.cpu().numpy().tolist() == ref_sum.tolist()
    assert top.cpu().numpy().tolist() == O.select_layers(A_dev, k).tolist()
    # the layers differ far more than the tolerance: the oracle's own scores rank them alike
    assert O.select_layers(A_oracle, k).tolist() == top.cpu().numpy().tolist()
