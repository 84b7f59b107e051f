"""Helpers shared by the GPU parity tests: device copies of synthetic workloads."""
import numpy as np
import torch

from paper_2608_26806_gb300 import avtp

# Score tolerance (bf16 inputs, fp32 accumulation) against the fp64 oracle.
RTOL = 1e-3
ATOL = 1e-5


def ensure_built():
    import __graft_entry__

    __graft_entry__.build()
    return avtp.load()


def bf16_dev(bits: np.ndarray, dev="cuda") -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).to(dev).view(torch.bfloat16)


def bits_of(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def dev_layout(lay, dev="cuda") -> avtp.Layout:
    return avtp.Layout.from_host(lay.cu_seqlens, lay.img_cu, lay.img_start, lay.img_len, device=dev)


class DevWorkload:
    def __init__(self, wl, dev="cuda"):
        self.wl = wl
        self.L = dev_layout(wl.layout, dev)
        self.t = {}
        for name in ("h_cur", "h_prior", "q", "k"):
            if name in wl.tensors:
                self.t[name] = bf16_dev(wl.tensors[name], dev)
        if "pos" in wl.tensors:
            self.t["pos"] = torch.from_numpy(wl.tensors["pos"]).to(dev)
        self.keep_ratio = torch.from_numpy(wl.keep_ratio).to(dev)

    def score_tensors(self, criterion):
        if criterion == "hidden_variation":
            return dict(h_cur=self.t["h_cur"], h_prior=self.t["h_prior"])
        return dict(q=self.t["q"], k=self.t["k"], softmax_scale=self.wl.softmax_scale)


def assert_scores_close(got: np.ndarray, ref: np.ndarray, mask: np.ndarray):
    np.testing.assert_allclose(got[mask], ref[mask], rtol=RTOL, atol=ATOL)


def near_tie(a: float, b: float) -> bool:
    """Oracle scores a and b are within the score tolerance of each other."""
    if np.isnan(a) or np.isnan(b):
        return np.isnan(a) and np.isnan(b)
    return abs(a - b) <= ATOL + RTOL * max(abs(a), abs(b))
