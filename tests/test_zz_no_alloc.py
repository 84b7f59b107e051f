"""avtp_select_noalloc: selection for callers that cannot allocate device memory.

Some callers of this library may not allocate GPU memory where they call it.
An inference engine may have reserved all free HBM for its KV-cache pool at
start-up and pass plugins nothing but their inputs and outputs. Code may also
run where allocation calls are not allowed. For them, avtp_select_noalloc
keeps its scratch in a fixed device array inside the library, instead of in
a caller workspace.

These tests call it through the C ABI, twice in a row on one stream with
different layouts. Each result must equal the workspace-based avtp_select and
the oracle's selection exactly: kept indices are integers, so the tolerance is
bit-exact, as for avtp_select itself. This file is named to be collected last;
it also passes on its own in a fresh process.
"""
import numpy as np
import pytest
import torch

from oracle import avtp_oracle as O
from paper_2608_26806_gb300 import avtp, synth
from tests.gpu_util import dev_layout, ensure_built

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    ensure_built()


def _case(segments, seed):
    """A layout, random scores with ties and NaN, random budgets and matching output offsets."""
    rng = np.random.default_rng(seed)
    lay = synth.Layout.from_segments(segments)
    T = lay.n_tokens
    sc = rng.standard_normal(T).astype(np.float32)
    sc[rng.random(T) < 0.1] = 0.5
    sc[rng.random(T) < 0.02] = np.nan
    budgets = np.array([int(rng.integers(0, v + 1)) for v in lay.img_len], dtype=np.int32)
    vis = lay.visual_mask()
    out_cu = np.zeros(lay.n_requests + 1, dtype=np.int32)
    for r in range(lay.n_requests):
        a, b = int(lay.cu_seqlens[r]), int(lay.cu_seqlens[r + 1])
        k = int(budgets[int(lay.img_cu[r]):int(lay.img_cu[r + 1])].sum())
        out_cu[r + 1] = out_cu[r] + k + int((~vis[a:b]).sum())
    L = dev_layout(lay)
    return dict(L=L, scores=torch.from_numpy(sc).cuda(), budgets=torch.from_numpy(budgets).cuda(),
                out_cu=torch.from_numpy(out_cu).cuda(), n_kept=int(out_cu[-1]),
                expected=O.select(lay, sc, budgets))


SEG_A = [[("t", 64)] + sum([[("t", 1), ("i", n), ("t", 1)] for n in (256, 1024, 640, 320, 900, 3000)], []) +
         [("t", 160)]]
SEG_B = [[("t", 7)], [("i", 5), ("t", 2), ("i", 1)], [("t", 3), ("i", 2049), ("t", 4)]]


def test_noalloc_select_matches_workspace_select_twice_in_a_row():
    cases = [_case(SEG_A, 1), _case(SEG_B, 2)]
    stream = torch.cuda.current_stream()
    got, status = [], []
    for c in cases:  # two calls in a row, ordered on one stream, no synchronisation between them
        kept = torch.full((c["n_kept"] + 8,), -7, dtype=torch.int32, device="cuda")
        st = torch.full((1,), -1, dtype=torch.int32, device="cuda")
        avtp.select_noalloc(c["L"], c["scores"], c["budgets"], c["out_cu"], kept, c["n_kept"], device_status=st,
                            stream=stream)
        got.append(kept)
        status.append(st)
    torch.cuda.synchronize()
    for c, kept, st in zip(cases, got, status):
        ref = avtp.select(c["L"], c["scores"], c["budgets"], c["out_cu"], c["n_kept"])
        torch.cuda.synchronize()
        assert int(st.item()) == avtp.OK
        assert torch.equal(kept[:c["n_kept"]].cpu(), ref.cpu())
        assert np.array_equal(kept[:c["n_kept"]].cpu().numpy(), c["expected"])
        assert torch.all(kept[c["n_kept"]:].cpu() == -7)  # nothing written past n_kept


def test_noalloc_select_rejects_layouts_above_its_fixed_limit():
    n = 16385  # one image more than AVTP_NOALLOC_MAX_IMAGES
    lay = synth.Layout.from_segments([[("i", 1)] * n])
    c = dict(L=dev_layout(lay), scores=torch.zeros(n, device="cuda"),
             budgets=torch.zeros(n, dtype=torch.int32, device="cuda"),
             out_cu=torch.tensor([0, 0], dtype=torch.int32, device="cuda"))
    kept = torch.empty(1, dtype=torch.int32, device="cuda")
    with pytest.raises(avtp.AVTPError) as e:
        avtp.select_noalloc(c["L"], c["scores"], c["budgets"], c["out_cu"], kept, 0)
    assert e.value.code == avtp.ERR_RANGE
