"""Thin Python binding of the AVTP C ABI (``include/avtp.h``).

Argument marshalling only: every step of the pruning stage runs in the CUDA
kernels of ``libavtp.so``. torch supplies device memory and streams. There is
no CPU fallback: if the library is missing or a call fails, this module raises.

Function names follow the C ABI (``score``, ``allocate``, ``select``,
``compact``, ``prune``, ``workspace_size``, ``kept_count_host``,
``read_device_status``); each takes torch tensors and calls the entry point of
the same name.
"""
from __future__ import annotations

import ctypes
import os
from ctypes import POINTER, c_float, c_int, c_int32, c_int64, c_size_t, c_void_p
from dataclasses import dataclass
from typing import Dict, Iterable, List, Optional, Sequence, Tuple

import numpy as np
import torch

from . import build as _build

OK = 0
ERR_INVALID_ARG = 1
ERR_UNSUPPORTED = 2
ERR_RANGE = 3
ERR_CUDA = 4
ERR_TIMEOUT = 5
ERR_DEVICE_INPUT = 6
ERR_WORKSPACE = 7

CRIT_HIDDEN_VARIATION = 0
CRIT_TEXT_ATTENTION = 1
MAX_ROW_SETS = 8
N_STEP_EVENTS = 5

_CRITERIA = {"hidden_variation": CRIT_HIDDEN_VARIATION, "text_attention": CRIT_TEXT_ATTENTION}
# avtp_query_set_t and avtp_attn_path_t
QUERIES_TEXT, QUERIES_LAST = 0, 1
PATH_AUTO, PATH_TENSOR, PATH_CUDA = 0, 1, 2
_QUERY_SETS = {"text": QUERIES_TEXT, "last": QUERIES_LAST}
_PATHS = {"auto": PATH_AUTO, "tensor": PATH_TENSOR, "cuda": PATH_CUDA}


class AVTPError(RuntimeError):
    """A non-OK status from the library: ``code`` (an avtp_status_t value) and the call it came from."""
    def __init__(self, code: int, where: str):
        self.code = int(code)
        super().__init__(f"{where}: {status_string(code)} (status {code})")


# ---------------------------------------------------------------- C structs
class _Layout(ctypes.Structure):
    _fields_ = [("n_requests", c_int32), ("n_images", c_int32), ("n_tokens", c_int64),
                ("cu_seqlens", c_void_p), ("img_cu", c_void_p), ("img_start", c_void_p), ("img_len", c_void_p)]


class _ScoreArgs(ctypes.Structure):
    _fields_ = [("criterion", c_int), ("h_cur", c_void_p), ("h_prior", c_void_p), ("hidden", c_int32),
                ("h_cur_stride", c_int64), ("h_prior_stride", c_int64), ("q", c_void_p), ("k", c_void_p),
                ("n_q_heads", c_int32), ("n_kv_heads", c_int32), ("head_dim", c_int32), ("q_stride", c_int64),
                ("k_stride", c_int64), ("softmax_scale", c_float), ("lse", c_void_p), ("lse_stride", c_int64),
                ("max_text_tokens", c_int64), ("query_set", c_int32), ("path", c_int32)]


class _AllocArgs(ctypes.Structure):
    _fields_ = [("keep_ratio", c_void_p), ("alpha", c_float), ("r_min", c_float), ("r_max", c_float),
                ("relative", c_int32)]


class _Rows(ctypes.Structure):
    _fields_ = [("in_", c_void_p), ("out", c_void_p), ("row_bytes", c_int64), ("in_stride", c_int64),
                ("out_stride", c_int64)]


class _ForwardArgs(ctypes.Structure):
    _fields_ = [("v", c_void_p), ("v_stride", c_int64), ("o", c_void_p), ("o_stride", c_int64), ("lse", c_void_p),
                ("lse_stride", c_int64)]


# ---------------------------------------------------------------- library
_LIB = None

# name -> (restype, argtypes); every symbol the header declares
SIGNATURES = {
    "avtp_workspace_size": (c_int, [POINTER(_Layout), POINTER(_ScoreArgs), POINTER(c_size_t)]),
    "avtp_score": (c_int, [POINTER(_Layout), POINTER(_ScoreArgs), c_void_p, c_void_p, c_void_p, c_size_t, c_void_p]),
    "avtp_forward_workspace_size": (c_int, [POINTER(_Layout), POINTER(_ScoreArgs), POINTER(_ForwardArgs),
                                            POINTER(c_size_t)]),
    "avtp_attn_forward": (c_int, [POINTER(_Layout), POINTER(_ScoreArgs), POINTER(_ForwardArgs), c_void_p, c_void_p,
                                  c_void_p, c_size_t, c_void_p]),
    "avtp_forward_timeline": (c_int, [c_void_p, c_int32]),
    "avtp_score_timeline": (c_int, [c_int32, c_void_p, c_int32]),
    "avtp_allocate": (c_int, [POINTER(_Layout), c_void_p, POINTER(_AllocArgs), c_void_p, c_void_p, c_void_p,
                              c_size_t, c_void_p]),
    "avtp_select": (c_int, [POINTER(_Layout), c_void_p, c_void_p, c_void_p, c_void_p, c_int64, c_void_p, c_size_t,
                            c_void_p]),
    "avtp_compact": (c_int, [c_void_p, c_int64, c_int64, POINTER(_Rows), c_int32, c_void_p, c_size_t, c_void_p]),
    "avtp_prune": (c_int, [POINTER(_Layout), POINTER(_ScoreArgs), POINTER(_AllocArgs), c_void_p, c_void_p, c_void_p,
                           c_void_p, c_void_p, c_int64, POINTER(_Rows), c_int32, c_void_p, c_size_t,
                           POINTER(c_void_p), c_void_p]),
    "avtp_select_noalloc": (c_int, [POINTER(_Layout), c_void_p, c_void_p, c_void_p, c_void_p, c_int64, c_void_p,
                                    c_void_p]),
    "avtp_kept_count_host": (c_int64, [c_void_p, c_void_p, c_void_p, c_void_p, c_int32]),
    "avtp_pruned_layout": (c_int, [POINTER(_Layout), c_void_p, c_void_p, c_void_p, c_void_p, c_size_t, c_void_p]),
    "avtp_kept_count_vis_host": (c_int64, [c_void_p, c_void_p, c_void_p, c_int32, c_void_p, c_void_p]),
    "avtp_wait_selftest": (c_int, [c_int64, c_int32, c_void_p, c_size_t, c_void_p]),
    "avtp_layer_attention": (c_int, [POINTER(_Layout), c_void_p, c_void_p, c_int32, c_int32, c_void_p, c_size_t,
                                     c_void_p]),
    "avtp_layer_select": (c_int, [c_void_p, c_int32, c_int32, c_int32, c_void_p, c_void_p, c_void_p]),
    "avtp_read_device_status": (c_int, [c_void_p, c_void_p, POINTER(c_int32)]),
    "avtp_status_string": (ctypes.c_char_p, [c_int32]),
    "avtp_version": (c_int32, []),
}


def library_path() -> str:
    """Path of the in-tree libavtp.so that ``load()`` opens: the diagnostic timeline build
    when the environment sets AVTP_TIMELINE=1, the normal build otherwise."""
    return _build.TIMELINE_LIB_PATH if os.environ.get("AVTP_TIMELINE") == "1" else _build.LIB_PATH


def load() -> ctypes.CDLL:
    """Load libavtp.so (built by ``__graft_entry__.build()``); raise if it is missing."""
    global _LIB
    if _LIB is not None:
        return _LIB
    path = library_path()
    if not os.path.exists(path):
        if os.environ.get("AVTP_AUTOBUILD") == "1":
            _build.build(timeline=path == _build.TIMELINE_LIB_PATH)
        else:
            raise RuntimeError(f"libavtp.so is not built ({path}); run __graft_entry__.build() first")
    lib = ctypes.CDLL(path)
    for name, (res, args) in SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _LIB = lib
    return lib


TIMELINE_EVENTS = ("prep_begin", "prep_end", "score_begin", "score_end", "select_begin", "select_dry_end",
                   "select_waited", "rule_begin", "rule_end", "select_end", "compact_begin", "compact_waited",
                   "compact_end", "hist_done")


def timeline(workspace: torch.Tensor) -> Dict[str, Tuple[int, int]]:
    """Phase stamps of the last avtp_prune on ``workspace`` (timeline build only): event ->
    (earliest, latest) global-timer nanoseconds over the CTAs that reached it; events no CTA
    reached are left out. Synchronises the device."""
    torch.cuda.synchronize()
    n = len(TIMELINE_EVENTS)
    raw = workspace[16:16 + 16 * n].cpu().numpy().view(np.uint64)
    out = {}
    for i, name in enumerate(TIMELINE_EVENTS):
        lo, hi = int(raw[i]), int(raw[n + i])
        if lo != 2 ** 64 - 1:
            out[name] = (lo, hi)
    return out


def status_string(code: int) -> str:
    """avtp_status_string: static English text for a status code."""
    return load().avtp_status_string(int(code)).decode()


def _check(code: int, where: str) -> None:
    if code != OK:
        raise AVTPError(code, where)


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    return None if t is None else int(t.data_ptr())


def _stream(stream) -> int:
    if stream is None:
        stream = torch.cuda.current_stream()
    return int(stream.cuda_stream) if hasattr(stream, "cuda_stream") else int(stream)


# ---------------------------------------------------------------- layout
@dataclass
class Layout:
    """A varlen-packed multi-image layout on the device (int32 tensors) plus host copies.

    A layout made by ``pruned_layout`` keeps its image spans on the device only: its
    host copy holds cu_seqlens, img_cu and the visual tokens per request (``n_vis``).
    """
    cu_seqlens: torch.Tensor
    img_cu: torch.Tensor
    img_start: torch.Tensor
    img_len: torch.Tensor
    host: Dict[str, np.ndarray]

    @staticmethod
    def from_host(cu_seqlens, img_cu, img_start, img_len, device="cuda") -> "Layout":
        """Copies host layout arrays (int32) to ``device`` and keeps the host copies."""
        host = {k: np.ascontiguousarray(np.asarray(v, dtype=np.int32))
                for k, v in dict(cu_seqlens=cu_seqlens, img_cu=img_cu, img_start=img_start, img_len=img_len).items()}
        dev = {k: torch.from_numpy(v.copy()).to(device) for k, v in host.items()}
        return Layout(host=host, **dev)

    @property
    def n_requests(self) -> int:
        """R, the number of varlen-packed requests."""
        return int(self.host["cu_seqlens"].shape[0] - 1)

    @property
    def n_images(self) -> int:
        """Images over all requests."""
        return int(self.host["img_cu"][-1])

    @property
    def n_tokens(self) -> int:
        """T, the packed tokens over all requests."""
        return int(self.host["cu_seqlens"][-1])

    @property
    def n_vis_per_request(self) -> np.ndarray:
        """Visual tokens of each request (int32 [R])."""
        if "n_vis" in self.host:
            return self.host["n_vis"]
        csum = np.concatenate([[0], np.cumsum(self.host["img_len"].astype(np.int64))])
        return (csum[self.host["img_cu"][1:]] - csum[self.host["img_cu"][:-1]]).astype(np.int32)

    @property
    def n_text(self) -> int:
        """Text tokens over all requests."""
        return self.n_tokens - int(self.n_vis_per_request.astype(np.int64).sum())

    def c(self) -> _Layout:
        """The avtp_layout_t the C calls take (pointers into the device tensors)."""
        return _Layout(self.n_requests, self.n_images, self.n_tokens, _ptr(self.cu_seqlens), _ptr(self.img_cu),
                       _ptr(self.img_start) if self.n_images else None, _ptr(self.img_len) if self.n_images else None)


def _score_args(criterion, h_cur=None, h_prior=None, q=None, k=None, softmax_scale=None, lse=None,
                max_text_tokens=0, query_set="text", path="auto") -> _ScoreArgs:
    a = _ScoreArgs()
    a.max_text_tokens = int(max_text_tokens)
    a.query_set = _QUERY_SETS[query_set] if isinstance(query_set, str) else int(query_set)
    a.path = _PATHS[path] if isinstance(path, str) else int(path)
    a.criterion = _CRITERIA[criterion] if isinstance(criterion, str) else int(criterion)
    if a.criterion == CRIT_HIDDEN_VARIATION:
        for t in (h_cur, h_prior):
            if t is None or t.dtype != torch.bfloat16 or t.dim() != 2 or t.stride(1) != 1:
                raise ValueError("h_cur / h_prior must be bf16 [T, hidden] with a contiguous last dim")
        a.h_cur, a.h_prior = _ptr(h_cur), _ptr(h_prior)
        a.hidden = h_cur.shape[1]
        a.h_cur_stride, a.h_prior_stride = h_cur.stride(0), h_prior.stride(0)
    else:
        for t in (q, k):
            if t is None or t.dtype != torch.bfloat16 or t.dim() != 3 or t.stride(2) != 1 or t.stride(1) != t.shape[2]:
                raise ValueError("q / k must be bf16 [T, heads, head_dim] with contiguous heads")
        a.q, a.k = _ptr(q), _ptr(k)
        a.n_q_heads, a.n_kv_heads, a.head_dim = q.shape[1], k.shape[1], q.shape[2]
        a.q_stride, a.k_stride = q.stride(0), k.stride(0)
        a.softmax_scale = float(softmax_scale if softmax_scale is not None else q.shape[2] ** -0.5)
        if lse is not None:
            if lse.dtype != torch.float32 or lse.dim() != 2 or lse.stride(1) != 1:
                raise ValueError("lse must be fp32 [Hq, T] with a contiguous last dim")
            a.lse, a.lse_stride = _ptr(lse), lse.stride(0)
    return a


def _alloc_args(keep_ratio: torch.Tensor, alpha=1.0, r_min=0.05, r_max=0.95, relative=False) -> _AllocArgs:
    if keep_ratio.dtype != torch.float32 or not keep_ratio.is_cuda:
        raise ValueError("keep_ratio must be a float32 CUDA tensor [R]")
    return _AllocArgs(_ptr(keep_ratio), float(alpha), float(r_min), float(r_max), 1 if relative else 0)


def _row_sets(rows: Sequence[Tuple[torch.Tensor, torch.Tensor]]) -> Tuple[ctypes.Array, int]:
    """(in, out) pairs gathered along dim 0: row j of out = row kept_idx[j] of in."""
    arr = (_Rows * MAX_ROW_SETS)()
    if len(rows) > MAX_ROW_SETS:
        raise ValueError(f"at most {MAX_ROW_SETS} row sets")
    for i, (src, dst) in enumerate(rows):
        es = src.element_size()
        row_elems = int(np.prod(src.shape[1:])) if src.dim() > 1 else 1
        if src.dim() > 1 and not src[0].is_contiguous():
            raise ValueError("each row must be contiguous")
        arr[i] = _Rows(_ptr(src), _ptr(dst), row_elems * es, src.stride(0) * es, dst.stride(0) * es)
    return arr, len(rows)


def workspace_size(layout: Layout, criterion=None, **score_tensors) -> int:
    """avtp_workspace_size: bytes of workspace a call needs for this layout and scoring setup."""
    lay = layout.c()
    sa = _score_args(criterion, max_text_tokens=layout.n_text, **score_tensors) if criterion is not None else None
    out = c_size_t()
    _check(load().avtp_workspace_size(ctypes.byref(lay), ctypes.byref(sa) if sa is not None else None,
                                      ctypes.byref(out)), "avtp_workspace_size")
    return int(out.value)


def new_workspace(nbytes: int, device="cuda") -> torch.Tensor:
    """A caller-owned workspace (torch allocations are 256-byte aligned)."""
    return torch.empty(max(int(nbytes), 256), dtype=torch.uint8, device=device)


# ---------------------------------------------------------------- entry points
def score(layout: Layout, criterion, *, h_cur=None, h_prior=None, q=None, k=None, softmax_scale=None, lse=None,
          query_set="text", path="auto", scores=None, img_sums=None, workspace=None, stream=None):
    """avtp_score: per-token scores (fp32 [T], text entries untouched) and fixed-point per-image sums.

    Text attention: ``query_set`` "text" (every text token) or "last" (the request's last
    token); ``path`` "auto", "tensor" (tcgen05) or "cuda" (CUDA cores)."""
    dev = layout.cu_seqlens.device
    sa = _score_args(criterion, h_cur, h_prior, q, k, softmax_scale, lse, max_text_tokens=layout.n_text,
                     query_set=query_set, path=path)
    if scores is None:
        scores = torch.zeros(layout.n_tokens, dtype=torch.float32, device=dev)
    if img_sums is None:
        img_sums = torch.empty(max(layout.n_images, 1), dtype=torch.int64, device=dev)
    if workspace is None:
        workspace = new_workspace(workspace_size(layout, criterion, h_cur=h_cur, h_prior=h_prior, q=q, k=k,
                                                 softmax_scale=softmax_scale, lse=lse, query_set=query_set,
                                                 path=path), dev)
    lay = layout.c()
    _check(load().avtp_score(ctypes.byref(lay), ctypes.byref(sa), _ptr(scores), _ptr(img_sums), _ptr(workspace),
                             workspace.numel(), _stream(stream)), "avtp_score")
    return scores, img_sums[:layout.n_images]


def _forward_args(v: torch.Tensor, o: torch.Tensor, lse: torch.Tensor) -> _ForwardArgs:
    if v.dtype != torch.bfloat16 or v.dim() != 3 or v.stride(2) != 1 or v.stride(1) != v.shape[2]:
        raise ValueError("v must be bf16 [T, Hkv, head_dim] with contiguous heads")
    if o.dtype != torch.float32 or o.dim() != 3 or o.stride(2) != 1 or o.stride(1) != o.shape[2]:
        raise ValueError("o must be fp32 [T, Hq, head_dim] with contiguous heads")
    if lse.dtype != torch.float32 or lse.dim() != 2 or lse.stride(1) != 1:
        raise ValueError("lse must be fp32 [Hq, T] with a contiguous last dim")
    return _ForwardArgs(_ptr(v), v.stride(0), _ptr(o), o.stride(0), _ptr(lse), lse.stride(0))


class ForwardCall:
    """A prepared avtp_attn_forward call: arguments marshalled once, outputs and workspace
    allocated once, so that ``run()`` is the C call alone (for timing and graphs)."""

    def __init__(self, layout: Layout, *, q, k, v, softmax_scale=None, scores: bool = True, query_set="text",
                 path="auto", o=None, lse=None, workspace=None):
        dev = layout.cu_seqlens.device
        T, Hq, d = q.shape
        self.layout = layout
        self.o = o if o is not None else torch.empty(T, Hq, d, dtype=torch.float32, device=dev)
        self.lse = lse if lse is not None else torch.empty(Hq, max(T, 1), dtype=torch.float32, device=dev)
        self.scores = torch.zeros(T, dtype=torch.float32, device=dev) if scores else None
        self.img_sums = torch.empty(max(layout.n_images, 1), dtype=torch.int64, device=dev) if scores else None
        self._keep = (q, k, v)
        self._sa = _score_args(CRIT_TEXT_ATTENTION, q=q, k=k, softmax_scale=softmax_scale,
                               max_text_tokens=layout.n_text, query_set=query_set, path=path)
        self._fa = _forward_args(v, self.o, self.lse)
        self._lay = layout.c()
        lib = load()
        if workspace is None:
            n = c_size_t()
            _check(lib.avtp_forward_workspace_size(ctypes.byref(self._lay), ctypes.byref(self._sa),
                                                   ctypes.byref(self._fa), ctypes.byref(n)),
                   "avtp_forward_workspace_size")
            workspace = new_workspace(int(n.value), dev)
        self.workspace = workspace

    def run(self, stream=None):
        _check(load().avtp_attn_forward(ctypes.byref(self._lay), ctypes.byref(self._sa), ctypes.byref(self._fa),
                                        _ptr(self.scores), _ptr(self.img_sums), _ptr(self.workspace),
                                        self.workspace.numel(), _stream(stream)), "avtp_attn_forward")
        return self


FORWARD_TIMELINE_SLOTS = ("top", "s_ready", "exchanged", "exp_done", "p_handed", "mma_s_entry", "mma_s_issued",
                          "mma_pv_entry", "mma_pv_ready", "mma_pv_issued")


def forward_timeline(n_blocks: int) -> np.ndarray:
    """avtp_forward_timeline: clock stamps int64 [n_blocks, 10] (FORWARD_TIMELINE_SLOTS) of the
    last forward call's first CTA; needs the timeline build (AVTP_TIMELINE=1)."""
    out = np.zeros((n_blocks, len(FORWARD_TIMELINE_SLOTS)), dtype=np.int64)
    _check(load().avtp_forward_timeline(out.ctypes.data, n_blocks), "avtp_forward_timeline")
    return out


SCORE_TIMELINE_SLOTS = ("load_issued", "mma_step", "mma_ready", "mma_issued", "acc_ready", "acc_released")


def score_timeline(pass_: int, n_steps: int) -> np.ndarray:
    """avtp_score_timeline: clock stamps int64 [n_steps, 6] (SCORE_TIMELINE_SLOTS) of the first
    CTA of criterion B's tensor-core pass 1 or 2; needs the timeline build (AVTP_TIMELINE=1)."""
    out = np.zeros((n_steps, len(SCORE_TIMELINE_SLOTS)), dtype=np.int64)
    _check(load().avtp_score_timeline(int(pass_), out.ctypes.data, n_steps), "avtp_score_timeline")
    return out


def attn_forward(layout: Layout, *, q, k, v, softmax_scale=None, scores: bool = True, query_set="text",
                 path="auto", stream=None):
    """avtp_attn_forward: the layer's causal attention forward, O (fp32 [T, Hq, d]) and the
    natural-log LSE (fp32 [Hq, T]), and with ``scores`` the text-attention scores and
    fixed-point image sums from that LSE. Returns (o, lse, scores, img_sums); the last
    two are None without ``scores``."""
    c = ForwardCall(layout, q=q, k=k, v=v, softmax_scale=softmax_scale, scores=scores, query_set=query_set,
                    path=path).run(stream)
    sums = c.img_sums[:layout.n_images] if c.img_sums is not None else None
    return c.o, c.lse[:, :layout.n_tokens], c.scores, sums


def allocate(layout: Layout, img_sums: torch.Tensor, keep_ratio: torch.Tensor, alpha=1.0, r_min=0.05, r_max=0.95,
             relative=False, budgets=None, out_cu_seqlens=None, workspace=None, stream=None):
    """avtp_allocate: per-image budgets (int32 [n_images]) and out_cu_seqlens (int32 [R+1])."""
    dev = layout.cu_seqlens.device
    aa = _alloc_args(keep_ratio, alpha, r_min, r_max, relative)
    if budgets is None:
        budgets = torch.empty(max(layout.n_images, 1), dtype=torch.int32, device=dev)
    if out_cu_seqlens is None:
        out_cu_seqlens = torch.empty(layout.n_requests + 1, dtype=torch.int32, device=dev)
    if workspace is None:
        workspace = new_workspace(workspace_size(layout), dev)
    lay = layout.c()
    _check(load().avtp_allocate(ctypes.byref(lay), _ptr(img_sums), ctypes.byref(aa), _ptr(budgets),
                                _ptr(out_cu_seqlens), _ptr(workspace), workspace.numel(), _stream(stream)),
           "avtp_allocate")
    return budgets[:layout.n_images], out_cu_seqlens


def select(layout: Layout, scores: torch.Tensor, budgets: torch.Tensor, out_cu_seqlens: torch.Tensor, n_kept: int,
           kept_idx=None, workspace=None, stream=None):
    """avtp_select: ascending packed positions of the kept tokens (int32 [n_kept])."""
    dev = layout.cu_seqlens.device
    if kept_idx is None:
        kept_idx = torch.empty(max(int(n_kept), 1), dtype=torch.int32, device=dev)
    if workspace is None:
        workspace = new_workspace(workspace_size(layout), dev)
    lay = layout.c()
    _check(load().avtp_select(ctypes.byref(lay), _ptr(scores), _ptr(budgets), _ptr(out_cu_seqlens), _ptr(kept_idx),
                              int(n_kept), _ptr(workspace), workspace.numel(), _stream(stream)), "avtp_select")
    return kept_idx[:int(n_kept)]


def select_noalloc(layout: Layout, scores: torch.Tensor, budgets: torch.Tensor, out_cu_seqlens: torch.Tensor,
                   kept_idx: torch.Tensor, n_kept: int, device_status: Optional[torch.Tensor] = None,
                   stream=None) -> torch.Tensor:
    """avtp_select_noalloc: avtp_select with the library's fixed scratch instead of a workspace.

    For callers that cannot allocate device memory at the call site; ``kept_idx``
    (int32, capacity >= n_kept) must be supplied by the caller.
    """
    lay = layout.c()
    _check(load().avtp_select_noalloc(ctypes.byref(lay), _ptr(scores), _ptr(budgets), _ptr(out_cu_seqlens),
                                      _ptr(kept_idx), int(n_kept), _ptr(device_status), _stream(stream)),
           "avtp_select_noalloc")
    return kept_idx[:int(n_kept)]


def compact(kept_idx: torch.Tensor, n_tokens: int, rows: Sequence[Tuple[torch.Tensor, torch.Tensor]],
            workspace=None, stream=None) -> None:
    """avtp_compact: for each (in, out) pair, out[j] = in[kept_idx[j]] along dim 0."""
    dev = kept_idx.device
    if workspace is None:
        workspace = new_workspace(256, dev)
    sets, n = _row_sets(rows)
    _check(load().avtp_compact(_ptr(kept_idx), kept_idx.numel(), int(n_tokens), sets, n, _ptr(workspace),
                               workspace.numel(), _stream(stream)), "avtp_compact")


def kept_count_vis_host(cu_seqlens: np.ndarray, n_vis: np.ndarray, keep_ratio: np.ndarray):
    """avtp_kept_count_vis_host: the pruned batch's size, host offsets and visual tokens per request."""
    cu = np.ascontiguousarray(np.asarray(cu_seqlens, dtype=np.int32))
    nv = np.ascontiguousarray(np.asarray(n_vis, dtype=np.int32))
    kr = np.ascontiguousarray(np.asarray(keep_ratio, dtype=np.float32))
    R = int(cu.shape[0] - 1)
    out_cu = np.zeros(R + 1, dtype=np.int32)
    out_nv = np.zeros(R, dtype=np.int32)
    n = load().avtp_kept_count_vis_host(cu.ctypes.data, nv.ctypes.data, kr.ctypes.data, R, out_cu.ctypes.data,
                                        out_nv.ctypes.data)
    if n < 0:
        raise AVTPError(ERR_INVALID_ARG, "avtp_kept_count_vis_host")
    return int(n), out_cu, out_nv


def pruned_layout(layout: Layout, keep_ratio_host: np.ndarray, budgets: torch.Tensor, out_cu_seqlens: torch.Tensor,
                  workspace=None, stream=None, into: Optional[Layout] = None) -> Layout:
    """avtp_pruned_layout: the layout of the batch that avtp_prune produced (device arrays).

    ``budgets`` and ``out_cu_seqlens`` are the prune call's device outputs; they are
    read on the device, so the pruned layout is usable in the same stream at once.
    ``into``: a layout returned by an earlier call whose device arrays are rewritten.
    """
    dev = layout.cu_seqlens.device
    NI = layout.n_images
    if into is not None:
        img_start, img_len = into.img_start, into.img_len
    else:
        img_start = torch.empty(max(NI, 1), dtype=torch.int32, device=dev)
        img_len = torch.empty(max(NI, 1), dtype=torch.int32, device=dev)
    if workspace is None:
        workspace = new_workspace(workspace_size(layout), dev)
    lay = layout.c()
    _check(load().avtp_pruned_layout(ctypes.byref(lay), _ptr(budgets), _ptr(img_start), _ptr(img_len),
                                     _ptr(workspace), workspace.numel(), _stream(stream)), "avtp_pruned_layout")
    if into is not None:
        return into
    _, cu_host, nv_host = kept_count_vis_host(layout.host["cu_seqlens"], layout.n_vis_per_request, keep_ratio_host)
    host = {"cu_seqlens": cu_host, "img_cu": layout.host["img_cu"].copy(), "n_vis": nv_host}
    return Layout(cu_seqlens=out_cu_seqlens[:layout.n_requests + 1], img_cu=layout.img_cu, img_start=img_start[:NI],
                  img_len=img_len[:NI], host=host)


def kept_count_host(layout_host: Dict[str, np.ndarray], keep_ratio: np.ndarray) -> int:
    """avtp_kept_count_host: sum_r floor(r_base*N_vis + 0.5) + N_txt over requests."""
    if "n_vis" in layout_host:  # a pruned layout: image lengths on the device only
        return kept_count_vis_host(layout_host["cu_seqlens"], layout_host["n_vis"], keep_ratio)[0]
    h = {k: np.ascontiguousarray(np.asarray(layout_host[k], dtype=np.int32))
         for k in ("cu_seqlens", "img_cu", "img_len")}
    kr = np.ascontiguousarray(np.asarray(keep_ratio, dtype=np.float32))
    img_len = h["img_len"] if h["img_len"].size else np.zeros(1, dtype=np.int32)
    n = load().avtp_kept_count_host(h["cu_seqlens"].ctypes.data, h["img_cu"].ctypes.data, img_len.ctypes.data,
                                    kr.ctypes.data, int(h["cu_seqlens"].shape[0] - 1))
    if n < 0:
        raise AVTPError(ERR_INVALID_ARG, "avtp_kept_count_host")
    return int(n)


def wait_selftest(limit_ns: int, arrive: bool, workspace: torch.Tensor, stream=None) -> None:
    """Runs the bounded-wait check kernel (``avtp_wait_selftest``); read the outcome
    with :func:`read_device_status` (``ERR_TIMEOUT`` when ``arrive`` is false)."""
    _check(load().avtp_wait_selftest(int(limit_ns), 1 if arrive else 0, _ptr(workspace),
                                     workspace.numel() * workspace.element_size(), _stream(stream)),
           "avtp_wait_selftest")


def layer_attention(layout: Layout, img_sums: torch.Tensor, A: torch.Tensor, layer: int, workspace=None,
                    stream=None) -> torch.Tensor:
    """avtp_layer_attention: column ``layer`` of A (int64 [R, n_layers]) <- each request's
    sum of text-attention image sums at that layer (pruning-layer selection, §3.3.2)."""
    if A.dtype != torch.int64 or A.dim() != 2 or not A.is_contiguous() or A.shape[0] != layout.n_requests:
        raise ValueError("A must be a contiguous int64 [R, n_layers] tensor")
    if workspace is None:
        workspace = new_workspace(workspace_size(layout), A.device)
    lay = layout.c()
    _check(load().avtp_layer_attention(ctypes.byref(lay), _ptr(img_sums), _ptr(A), A.shape[1], int(layer),
                                       _ptr(workspace), workspace.numel(), _stream(stream)), "avtp_layer_attention")
    return A


def layer_select(A: torch.Tensor, k: int, stream=None) -> Tuple[torch.Tensor, torch.Tensor]:
    """avtp_layer_select: (rank_sum int64 [n_layers], top_layers int32 [k]) from A [N, n_layers]."""
    if A.dtype != torch.int64 or A.dim() != 2 or not A.is_contiguous():
        raise ValueError("A must be a contiguous int64 [n_samples, n_layers] tensor")
    rank_sum = torch.empty(A.shape[1], dtype=torch.int64, device=A.device)
    top = torch.empty(int(k), dtype=torch.int32, device=A.device)
    _check(load().avtp_layer_select(_ptr(A), A.shape[0], A.shape[1], int(k), _ptr(rank_sum), _ptr(top),
                                    _stream(stream)), "avtp_layer_select")
    return rank_sum, top


def read_device_status(workspace: torch.Tensor, stream=None) -> int:
    """avtp_read_device_status: waits for ``stream`` and returns the workspace's status word."""
    out = c_int32()
    _check(load().avtp_read_device_status(_ptr(workspace), _stream(stream), ctypes.byref(out)),
           "avtp_read_device_status")
    return int(out.value)


@dataclass
class PruneBuffers:
    """Every buffer one avtp_prune call touches, allocated once for a fixed layout."""
    scores: torch.Tensor
    img_sums: torch.Tensor
    budgets: torch.Tensor
    out_cu_seqlens: torch.Tensor
    kept_idx: torch.Tensor
    workspace: torch.Tensor
    outputs: Dict[str, torch.Tensor]
    n_kept: int


def prune_buffers(layout: Layout, keep_ratio_host: np.ndarray, criterion, score_tensors: Dict[str, torch.Tensor],
                  rows: Dict[str, torch.Tensor], planes: Dict[str, torch.Tensor]) -> PruneBuffers:
    """Every output buffer and the workspace of an avtp_prune call, sized on the host (no device read)."""
    dev = layout.cu_seqlens.device
    n_kept = kept_count_host(layout.host, keep_ratio_host)
    outputs = {}
    for name, src in rows.items():
        outputs[name] = torch.empty((n_kept,) + tuple(src.shape[1:]), dtype=src.dtype, device=dev)
    for name, src in planes.items():
        outputs[name] = torch.empty((src.shape[0], n_kept), dtype=src.dtype, device=dev)
    ws = new_workspace(workspace_size(layout, criterion, **score_tensors), dev)
    return PruneBuffers(
        scores=torch.zeros(layout.n_tokens, dtype=torch.float32, device=dev),
        img_sums=torch.empty(max(layout.n_images, 1), dtype=torch.int64, device=dev),
        budgets=torch.empty(max(layout.n_images, 1), dtype=torch.int32, device=dev),
        out_cu_seqlens=torch.empty(layout.n_requests + 1, dtype=torch.int32, device=dev),
        kept_idx=torch.empty(max(n_kept, 1), dtype=torch.int32, device=dev),
        workspace=ws, outputs=outputs, n_kept=n_kept)


class PruneCall:
    """A prepared avtp_prune call: C structs built once, then launched with ``run()``.

    ``rows``: name -> [T, ...] tensors gathered along dim 0; ``planes``: name ->
    [P, T] tensors (e.g. M-RoPE position ids) gathered along dim 1.
    """

    def __init__(self, layout: Layout, criterion, *, keep_ratio: torch.Tensor, keep_ratio_host: np.ndarray,
                 alpha=1.0, r_min=0.05, r_max=0.95, relative=None, rows: Optional[Dict[str, torch.Tensor]] = None,
                 planes: Optional[Dict[str, torch.Tensor]] = None, buffers: Optional[PruneBuffers] = None,
                 **score_tensors):
        rows = rows or {}
        planes = planes or {}
        if relative is None:
            crit = _CRITERIA[criterion] if isinstance(criterion, str) else int(criterion)
            relative = crit == CRIT_TEXT_ATTENTION
        self.layout = layout
        self.buffers = buffers or prune_buffers(layout, keep_ratio_host, criterion, score_tensors, rows, planes)
        b = self.buffers
        self._lay = layout.c()
        self._sa = _score_args(criterion, max_text_tokens=layout.n_text, **score_tensors)
        self._aa = _alloc_args(keep_ratio, alpha, r_min, r_max, relative)
        pairs: List[Tuple[torch.Tensor, torch.Tensor]] = []
        for name, src in rows.items():
            pairs.append((src, b.outputs[name]))
        for name, src in planes.items():
            for p in range(src.shape[0]):
                pairs.append((src[p], b.outputs[name][p]))
        self._sets, self._n_sets = _row_sets(pairs)
        self._keep_alive = (keep_ratio, rows, planes, score_tensors)

    def run(self, stream=None, step_events: Optional[Sequence] = None) -> PruneBuffers:
        """Launches the prepared avtp_prune call on ``stream``; ``step_events`` (5 CUDA events) times its steps."""
        b = self.buffers
        ev = None
        if step_events is not None:  # 5 events: start, after validation, scoring, allocation+selection, compaction
            if len(step_events) != N_STEP_EVENTS:
                raise ValueError(f"step_events needs {N_STEP_EVENTS} events")
            ev = (c_void_p * N_STEP_EVENTS)(*[int(e.cuda_event) if hasattr(e, "cuda_event") else int(e)
                                              for e in step_events])
        _check(load().avtp_prune(ctypes.byref(self._lay), ctypes.byref(self._sa), ctypes.byref(self._aa),
                                 _ptr(b.scores), _ptr(b.img_sums), _ptr(b.budgets), _ptr(b.out_cu_seqlens),
                                 _ptr(b.kept_idx), b.n_kept, self._sets, self._n_sets, _ptr(b.workspace),
                                 b.workspace.numel(), ev, _stream(stream)), "avtp_prune")
        return b


def prune(layout: Layout, criterion, *, keep_ratio: torch.Tensor, keep_ratio_host: np.ndarray, alpha=1.0,
          r_min=0.05, r_max=0.95, relative=None, rows=None, planes=None, stream=None, **score_tensors) -> PruneBuffers:
    """avtp_prune: score -> allocate -> select -> compact in one call on one stream."""
    call = PruneCall(layout, criterion, keep_ratio=keep_ratio, keep_ratio_host=keep_ratio_host, alpha=alpha,
                     r_min=r_min, r_max=r_max, relative=relative, rows=rows, planes=planes, **score_tensors)
    return call.run(stream)
