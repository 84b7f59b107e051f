"""Seeded synthetic inputs for the AVTP pruning stage.

This module draws token layouts, per-image signal strengths, keep ratios and the
bf16 tensors (q, k, h_prior, h_cur, pos) that both the CUDA path and the CPU
oracle read. It holds none of the pruning arithmetic: no score, no budget, no
selection. Everything here is input construction.

The five named workloads are multi-image LVLM prefill shapes (LLaVA-OneVision-7B,
Qwen3-VL-8B, InternVL3.5-8B, a long stress case and a tiny case). They stand in
for the multi-image benchmarks the paper evaluates on (MuirBench, MIRB, BLINK,
Q-Bench2, NLVR2; paper §4.1), whose data and model weights are not used here:
the pruning stage only sees tensors of these shapes.

Conventions
-----------
* bf16 tensors are numpy ``uint16`` arrays holding bf16 bit patterns, obtained
  from fp32 N(0,1) draws by round-to-nearest-even.
* A layout is varlen-packed: request r owns packed tokens
  ``[cu_seqlens[r], cu_seqlens[r+1])``; its images are entries
  ``img_cu[r] .. img_cu[r+1]-1`` of ``img_start`` / ``img_len``, whose spans are
  request-local, sorted and disjoint. Tokens outside every span are text.
* Each tensor draws from its own child of ``SeedSequence(seed)``, so generating
  only the criterion-A tensors does not shift the criterion-B streams.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Dict, List, Optional, Sequence, Tuple

import numpy as np
import torch

CONFIG_NAMES = ("tiny", "llava_ov_7b", "qwen3_vl_8b", "internvl3_5_8b", "long")
BASE_SEED = 20260
_CHUNK_ROWS = 4096


# ----------------------------------------------------------------------------
# bf16 helpers (format conversion only)
# ----------------------------------------------------------------------------
def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round finite fp32 values to bf16 (nearest, ties to even); return the bits.

    torch's CPU cast is used only because it is fast and multi-threaded; it rounds
    to nearest-even like the bit recipe ``(u + 0x7FFF + ((u >> 16) & 1)) >> 16``.
    """
    x = np.ascontiguousarray(x, dtype=np.float32)
    return torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    """Widen bf16 bit patterns to fp32 (exact)."""
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


# ----------------------------------------------------------------------------
# Layout
# ----------------------------------------------------------------------------
@dataclass
class Layout:
    cu_seqlens: np.ndarray  # int32 [R+1]
    img_cu: np.ndarray      # int32 [R+1]
    img_start: np.ndarray   # int32 [n_img], request-local
    img_len: np.ndarray     # int32 [n_img]

    @property
    def n_requests(self) -> int:
        return int(self.cu_seqlens.shape[0] - 1)

    @property
    def n_images(self) -> int:
        return int(self.img_len.shape[0])

    @property
    def n_tokens(self) -> int:
        return int(self.cu_seqlens[-1])

    def request_of_image(self) -> np.ndarray:
        req = np.zeros(self.n_images, dtype=np.int64)
        for r in range(self.n_requests):
            req[self.img_cu[r]:self.img_cu[r + 1]] = r
        return req

    def visual_mask(self) -> np.ndarray:
        """Boolean [T]: True where the packed token lies inside an image span."""
        m = np.zeros(self.n_tokens, dtype=bool)
        for r in range(self.n_requests):
            base = int(self.cu_seqlens[r])
            for i in range(int(self.img_cu[r]), int(self.img_cu[r + 1])):
                s = base + int(self.img_start[i])
                m[s:s + int(self.img_len[i])] = True
        return m

    def n_visual_per_request(self) -> np.ndarray:
        out = np.zeros(self.n_requests, dtype=np.int64)
        for r in range(self.n_requests):
            out[r] = int(self.img_len[self.img_cu[r]:self.img_cu[r + 1]].sum())
        return out

    @staticmethod
    def from_segments(requests: Sequence[Sequence[Tuple[str, int]]]) -> "Layout":
        """Build a layout from per-request runs, e.g. ``[[("t", 8), ("i", 64), ("t", 4)]]``.

        ``"t"`` adds a run of text tokens, ``"i"`` one image of that many tokens.
        """
        cu = [0]
        img_cu = [0]
        starts: List[int] = []
        lens: List[int] = []
        for req in requests:
            pos = 0
            for kind, n in req:
                if kind == "i":
                    starts.append(pos)
                    lens.append(int(n))
                elif kind != "t":
                    raise ValueError(f"unknown run kind {kind!r}")
                pos += int(n)
            cu.append(cu[-1] + pos)
            img_cu.append(len(lens))
        return Layout(
            cu_seqlens=np.asarray(cu, dtype=np.int32),
            img_cu=np.asarray(img_cu, dtype=np.int32),
            img_start=np.asarray(starts, dtype=np.int32),
            img_len=np.asarray(lens, dtype=np.int32),
        )


# ----------------------------------------------------------------------------
# Workload
# ----------------------------------------------------------------------------
@dataclass
class Workload:
    name: str
    layout: Layout
    keep_ratio: np.ndarray        # float32 [R]
    signal: np.ndarray            # float32 [n_img]: per-image signal used to build inputs
    hidden: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    pos_planes: int
    seed: int
    # paper hyper-parameters (alpha = 1.0 and clamps [5%, 95%])
    alpha: float = 1.0
    r_min: float = 0.05
    r_max: float = 0.95
    tensors: Dict[str, np.ndarray] = field(default_factory=dict)

    @property
    def n_tokens(self) -> int:
        return self.layout.n_tokens

    @property
    def softmax_scale(self) -> float:
        return float(np.float32(1.0 / np.sqrt(self.head_dim)))

    def __getattr__(self, item):
        t = self.__dict__.get("tensors")
        if t is not None and item in t:
            return t[item]
        raise AttributeError(item)


def _layout_for(name: str, rng: np.random.Generator):
    """Token layout, per-image signal and per-request keep ratio for a named config."""
    if name == "tiny":
        lay = Layout.from_segments([[("i", 64), ("i", 64), ("i", 64), ("t", 32)]])
        sig = np.array([0.0, 0.5, 1.0], dtype=np.float32)
        kr = np.array([0.5], dtype=np.float32)
        dims = (256, 4, 2, 64, 1)
    elif name == "llava_ov_7b":
        lay = Layout.from_segments([[("t", 8), ("i", 729)] * 8 + [("t", 64)]])
        sig = rng.uniform(0.0, 1.0, size=8).astype(np.float32)
        kr = np.array([0.25], dtype=np.float32)
        dims = (3584, 28, 4, 128, 1)
    elif name == "qwen3_vl_8b":
        counts = rng.integers(0, 13, size=16) * 64 + 256  # {256, 320, ..., 1024}
        segs = [("t", 64)]
        for n in counts:
            segs += [("t", 1), ("i", int(n)), ("t", 1)]
        segs.append(("t", 160))
        lay = Layout.from_segments([segs])
        a = rng.lognormal(0.0, 1.0, size=16)
        sig = (a / a.max()).astype(np.float32)
        kr = np.array([0.33], dtype=np.float32)
        dims = (4096, 32, 8, 128, 3)
    elif name == "internvl3_5_8b":
        m = rng.integers(4, 33, size=8)
        t = rng.integers(64, 513, size=8)
        reqs = []
        for r in range(8):
            segs = []
            for _ in range(int(m[r])):
                segs += [("t", 1), ("i", 256), ("t", 1)]
            segs.append(("t", int(t[r] - 2 * m[r])))
            reqs.append(segs)
        lay = Layout.from_segments(reqs)
        sig = rng.uniform(0.0, 1.0, size=lay.n_images).astype(np.float32)
        kr = rng.choice(np.array([0.25, 0.33, 0.5], dtype=np.float32), size=8).astype(np.float32)
        dims = (4096, 32, 8, 128, 1)
    elif name == "long":
        reqs = []
        for _ in range(4):
            segs = []
            for _ in range(64):
                segs += [("t", 1), ("i", 1024), ("t", 1)]
            segs.append(("t", 384))
            reqs.append(segs)
        lay = Layout.from_segments(reqs)
        sig = np.full(lay.n_images, 0.1, dtype=np.float32)
        for r in range(4):
            hot = rng.choice(64, size=2, replace=False)
            sig[r * 64 + hot] = 2.0
        kr = np.array([0.125] * 4, dtype=np.float32)
        dims = (4096, 32, 8, 128, 1)
    else:
        raise KeyError(f"unknown config {name!r}; known: {CONFIG_NAMES}")
    return lay, sig, kr, dims


def _normal_bf16(rng: np.random.Generator, rows: int, cols: int) -> np.ndarray:
    out = np.empty((rows, cols), dtype=np.uint16)
    for r0 in range(0, rows, _CHUNK_ROWS):
        r1 = min(rows, r0 + _CHUNK_ROWS)
        out[r0:r1] = f32_to_bf16_bits(rng.standard_normal((r1 - r0, cols), dtype=np.float32))
    return out


def _row_signal(layout: Layout, signal: np.ndarray, text_value: float, offset: float) -> np.ndarray:
    """Per packed token: offset + signal of its image, or text_value on text."""
    out = np.full(layout.n_tokens, text_value, dtype=np.float32)
    for r in range(layout.n_requests):
        base = int(layout.cu_seqlens[r])
        for i in range(int(layout.img_cu[r]), int(layout.img_cu[r + 1])):
            s = base + int(layout.img_start[i])
            out[s:s + int(layout.img_len[i])] = offset + float(signal[i])
    return out


def build_tensors(wl: Workload, parts: Sequence[str] = ("A", "B", "pos")) -> Workload:
    """Draw the tensors of ``wl`` for the requested criteria.

    ``"A"``: ``h_prior`` = N(0,1) and ``h_cur`` = h_prior + beta * Z with beta = 0.25 on
    text and 0.25 + signal_i on image i (bf16 [T, D]).
    ``"B"``: ``q`` [T, Hq, d] and ``k`` [T, Hkv, d] N(0,1); keys of image i are shifted
    by signal_i times the mean query of their KV group over the request's text rows.
    ``"V"``: ``v`` [T, Hkv, d] N(0,1), the values of the layer's attention forward.
    ``"pos"``: int32 [P, T] with pos[p, t] = t + p*T (distinct per plane).
    """
    lay = wl.layout
    T = lay.n_tokens
    # child i of a fresh seed sequence is the same whatever the number spawned, so the
    # values' stream (child 5) leaves the other tensors unchanged
    children = np.random.SeedSequence(wl.seed).spawn(6)
    if "A" in parts:
        rng_p = np.random.default_rng(children[3])
        rng_z = np.random.default_rng(children[4])
        h_prior = _normal_bf16(rng_p, T, wl.hidden)
        beta = _row_signal(lay, wl.signal, 0.25, 0.25)
        h_cur = np.empty_like(h_prior)
        for r0 in range(0, T, _CHUNK_ROWS):
            r1 = min(T, r0 + _CHUNK_ROWS)
            z = rng_z.standard_normal((r1 - r0, wl.hidden), dtype=np.float32)
            hc = bf16_bits_to_f32(h_prior[r0:r1]) + beta[r0:r1, None] * z
            h_cur[r0:r1] = f32_to_bf16_bits(hc)
        wl.tensors["h_prior"] = h_prior
        wl.tensors["h_cur"] = h_cur
    if "B" in parts:
        rng_q = np.random.default_rng(children[1])
        rng_k = np.random.default_rng(children[2])
        Hq, Hkv, d = wl.n_q_heads, wl.n_kv_heads, wl.head_dim
        q = _normal_bf16(rng_q, T, Hq * d).reshape(T, Hq, d)
        k32 = np.empty((T, Hkv, d), dtype=np.uint16)
        vis = lay.visual_mask()
        grp = Hq // Hkv
        for r0 in range(0, T, _CHUNK_ROWS):
            r1 = min(T, r0 + _CHUNK_ROWS)
            k32[r0:r1] = _normal_bf16(rng_k, r1 - r0, Hkv * d).reshape(r1 - r0, Hkv, d)
        for r in range(lay.n_requests):
            a, b = int(lay.cu_seqlens[r]), int(lay.cu_seqlens[r + 1])
            text_rows = np.nonzero(~vis[a:b])[0] + a
            if text_rows.size == 0:
                continue
            qt = bf16_bits_to_f32(q[text_rows]).astype(np.float64)  # [nt, Hq, d]
            mean_q = qt.reshape(-1, Hkv, grp, d).mean(axis=(0, 2)).astype(np.float32)  # [Hkv, d]
            for i in range(int(lay.img_cu[r]), int(lay.img_cu[r + 1])):
                s = a + int(lay.img_start[i])
                e = s + int(lay.img_len[i])
                kf = bf16_bits_to_f32(k32[s:e]) + np.float32(wl.signal[i]) * mean_q[None]
                k32[s:e] = f32_to_bf16_bits(kf)
        wl.tensors["q"] = q
        wl.tensors["k"] = k32
    if "V" in parts:
        rng_v = np.random.default_rng(children[5])
        Hkv, d = wl.n_kv_heads, wl.head_dim
        v = np.empty((T, Hkv, d), dtype=np.uint16)
        for r0 in range(0, T, _CHUNK_ROWS):
            r1 = min(T, r0 + _CHUNK_ROWS)
            v[r0:r1] = _normal_bf16(rng_v, r1 - r0, Hkv * d).reshape(r1 - r0, Hkv, d)
        wl.tensors["v"] = v
    if "pos" in parts:
        P = wl.pos_planes
        pos = (np.arange(T, dtype=np.int64)[None, :] + np.arange(P, dtype=np.int64)[:, None] * T)
        wl.tensors["pos"] = pos.astype(np.int32)
    return wl


def make_workload(name: str, parts: Sequence[str] = ("A", "B", "pos"), seed: Optional[int] = None) -> Workload:
    """Build one of the five named workloads with seed ``20260 + config index``."""
    idx = CONFIG_NAMES.index(name)
    seed = BASE_SEED + idx if seed is None else int(seed)
    children = np.random.SeedSequence(seed).spawn(5)
    rng_layout = np.random.default_rng(children[0])
    lay, sig, kr, (D, Hq, Hkv, d, P) = _layout_for(name, rng_layout)
    wl = Workload(name=name, layout=lay, keep_ratio=kr, signal=sig, hidden=D, n_q_heads=Hq,
                  n_kv_heads=Hkv, head_dim=d, pos_planes=P, seed=seed)
    return build_tensors(wl, parts)


def make_custom(requests: Sequence[Sequence[Tuple[str, int]]], *, hidden: int = 64, n_q_heads: int = 4,
                n_kv_heads: int = 2, head_dim: int = 64, keep_ratio=0.5, signal=None, seed: int = 7,
                pos_planes: int = 1, parts: Sequence[str] = ("A", "B", "pos")) -> Workload:
    """A small workload on a hand-written layout (for edge-case tests)."""
    lay = Layout.from_segments(requests)
    rng = np.random.default_rng(seed)
    if signal is None:
        signal = rng.uniform(0.0, 1.0, size=lay.n_images)
    kr = np.broadcast_to(np.asarray(keep_ratio, dtype=np.float32), (lay.n_requests,)).copy()
    wl = Workload(name="custom", layout=lay, keep_ratio=kr, signal=np.asarray(signal, dtype=np.float32),
                  hidden=hidden, n_q_heads=n_q_heads, n_kv_heads=n_kv_heads, head_dim=head_dim,
                  pos_planes=pos_planes, seed=seed)
    return build_tensors(wl, parts)
