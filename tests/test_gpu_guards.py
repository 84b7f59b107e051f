"""Out-of-bounds writes, caught without a sanitizer: every buffer a call writes is
carved from a larger allocation whose guard regions on both sides hold a known byte
pattern, and the guards are compared after the call. The results must still equal the
unguarded run's (and so the oracle's, which the parity tests check)."""
import numpy as np
import pytest
import torch

from paper_2608_26806_gb300 import avtp, synth
from tests.gpu_util import DevWorkload, ensure_built

pytestmark = pytest.mark.gpu

GUARD = 4096     # bytes on each side; keeps the 256-byte alignment of workspaces
PATTERN = 0xA5


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    ensure_built()


class Guarded:
    def __init__(self):
        self.bases = []

    def __call__(self, shape, dtype):
        n = int(np.prod(shape)) if len(shape) else 1
        nbytes = n * torch.empty((), dtype=dtype).element_size()
        base = torch.full((GUARD + nbytes + GUARD,), PATTERN, dtype=torch.uint8, device="cuda")
        self.bases.append((base, nbytes))
        return base[GUARD:GUARD + nbytes].view(dtype).view(shape)

    def intact(self):
        torch.cuda.synchronize()
        for base, nbytes in self.bases:
            head, tail = base[:GUARD], base[GUARD + nbytes:]
            if not (bool((head == PATTERN).all()) and bool((tail == PATTERN).all())):
                return False
        return True


_CASES = {
    "tiny": None,
    "qwen3_vl_8b": None,
    "ragged": [[("t", 3), ("i", 3000), ("t", 1), ("i", 1), ("i", 129), ("t", 5)],
               [("i", 700), ("t", 2), ("i", 256), ("i", 257)], [("t", 9)]],
}


def _workload(case):
    if _CASES[case] is None:
        return synth.make_workload(case)
    return synth.make_custom(_CASES[case], keep_ratio=0.3, n_q_heads=8, n_kv_heads=2, head_dim=128, hidden=256)


@pytest.mark.parametrize("case", sorted(_CASES))
@pytest.mark.parametrize("criterion", ["hidden_variation", "text_attention"])
def test_fused_stage_writes_nothing_outside_its_buffers(case, criterion):
    wl = _workload(case)
    dw = DevWorkload(wl)
    lay = wl.layout
    T, NI, R = lay.n_tokens, lay.n_images, lay.n_requests
    kw = dw.score_tensors(criterion)
    ref = avtp.prune(dw.L, criterion, keep_ratio=dw.keep_ratio, keep_ratio_host=wl.keep_ratio,
                     rows={"hidden": dw.t["h_cur"]}, planes={"pos": dw.t["pos"]}, **kw)
    torch.cuda.synchronize()
    n_kept = ref.n_kept
    g = Guarded()
    bufs = avtp.PruneBuffers(
        scores=g((T,), torch.float32), img_sums=g((NI,), torch.int64), budgets=g((NI,), torch.int32),
        out_cu_seqlens=g((R + 1,), torch.int32), kept_idx=g((n_kept,), torch.int32),
        workspace=g((avtp.workspace_size(dw.L, criterion, **kw),), torch.uint8),
        outputs={"hidden": g((n_kept, wl.hidden), torch.bfloat16),
                 "pos": g(tuple(dw.t["pos"].shape[:1]) + (n_kept,), dw.t["pos"].dtype)},
        n_kept=n_kept)
    bufs.scores.zero_()
    call = avtp.PruneCall(dw.L, criterion, keep_ratio=dw.keep_ratio, keep_ratio_host=wl.keep_ratio,
                          rows={"hidden": dw.t["h_cur"]}, planes={"pos": dw.t["pos"]}, buffers=bufs, **kw)
    for _ in range(2):  # the second call reuses the workspace as a serving loop would
        call.run()
    assert g.intact()
    assert avtp.read_device_status(bufs.workspace) == avtp.OK
    vis = lay.visual_mask()
    assert torch.equal(bufs.scores[torch.from_numpy(vis).cuda()], ref.scores[torch.from_numpy(vis).cuda()])
    for name in ("img_sums", "budgets"):
        assert torch.equal(getattr(bufs, name), getattr(ref, name)[:NI])
    assert torch.equal(bufs.out_cu_seqlens, ref.out_cu_seqlens)
    assert torch.equal(bufs.kept_idx, ref.kept_idx[:n_kept])
    for name in ("hidden", "pos"):
        assert torch.equal(bufs.outputs[name], ref.outputs[name])


@pytest.mark.parametrize("case", ["qwen3_vl_8b", "ragged"])
def test_single_steps_write_nothing_outside_their_buffers(case):
    wl = _workload(case)
    dw = DevWorkload(wl)
    lay = wl.layout
    T, NI, R = lay.n_tokens, lay.n_images, lay.n_requests
    g = Guarded()
    kw = dw.score_tensors("text_attention")
    ws = g((avtp.workspace_size(dw.L, "text_attention", **kw),), torch.uint8)
    scores = g((T,), torch.float32)
    scores.zero_()
    sums = g((NI,), torch.int64)
    avtp.score(dw.L, "text_attention", scores=scores, img_sums=sums, workspace=ws, **kw)
    budgets, out_cu = g((NI,), torch.int32), g((R + 1,), torch.int32)
    avtp.allocate(dw.L, sums, dw.keep_ratio, relative=True, budgets=budgets, out_cu_seqlens=out_cu, workspace=ws)
    n_kept = avtp.kept_count_host(dw.L.host, wl.keep_ratio)
    kept = g((n_kept,), torch.int32)
    avtp.select(dw.L, scores, budgets, out_cu, n_kept, kept_idx=kept, workspace=ws)
    hidden = g((n_kept, wl.hidden), torch.bfloat16)
    avtp.compact(kept, T, [(dw.t["h_cur"], hidden)], workspace=ws)
    assert g.intact()
    assert avtp.read_device_status(ws) == avtp.OK
    assert int(out_cu[-1].item()) == n_kept
    assert torch.equal(hidden, dw.t["h_cur"][kept.long()])
