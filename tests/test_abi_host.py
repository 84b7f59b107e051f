"""C ABI checks that need no GPU: the library loads, exports every symbol that
include/avtp.h declares, and its host-side logic (argument validation, output
sizing, status strings) behaves as documented. No call here reaches a kernel:
every invalid-argument path returns before the first CUDA call.
"""
import ctypes
import os
import re
import shutil
import subprocess

import numpy as np
import pytest

from oracle import avtp_oracle as O
from paper_2608_26806_gb300 import avtp, synth
from tests.gpu_util import ensure_built

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "avtp.h")


@pytest.fixture(scope="module")
def lib():
    return ensure_built()


def declared_functions():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"AVTP_API\s+[\w\s\*]+?\b(avtp_\w+)\s*\(", text)))


def test_header_declares_the_stage_entry_points():
    names = declared_functions()
    for required in ("avtp_score", "avtp_allocate", "avtp_select", "avtp_compact", "avtp_prune"):
        assert required in names


def test_library_exports_every_declared_symbol(lib):
    out = subprocess.run(["nm", "-D", "--defined-only", avtp.library_path()], capture_output=True, text=True,
                         check=True).stdout
    exported = set(re.findall(r"\bT\s+(avtp_\w+)", out))
    for name in declared_functions():
        assert name in exported, name
        assert hasattr(lib, name)
        assert name in avtp.SIGNATURES  # the binding wraps each one


def _c_type_matches(c_type: str, ct) -> bool:
    c_type = " ".join(c_type.replace("const", " ").split())
    if "*" in c_type or c_type == "avtp_stream_t":
        return ct in (ctypes.c_void_p, ctypes.c_char_p) or (isinstance(ct, type) and issubclass(ct, ctypes._Pointer))
    return {"int64_t": ctypes.c_int64, "int32_t": ctypes.c_int32, "size_t": ctypes.c_size_t,
            "avtp_status_t": ctypes.c_int, "int": ctypes.c_int}.get(c_type.split()[0]) is ct


def test_binding_signatures_match_the_header():
    # every argument of every declared call: same count, and pointer / integer width alike
    text = open(HEADER).read()
    decls = re.findall(r"AVTP_API\s+([\w\s\*]+?)\b(avtp_\w+)\s*\(([^;]*?)\)\s*;", text, re.S)
    assert len(decls) == len(declared_functions())
    for ret, name, params in decls:
        res, args = avtp.SIGNATURES[name]
        plist = [] if params.strip() in ("", "void") else [p.strip() for p in params.split(",")]
        assert len(plist) == len(args), name
        for p, ct in zip(plist, args):
            c_type = re.sub(r"\b\w+$", "", p).strip() if "*" not in p.split()[-1] else p
            c_type = p[:p.rfind("*") + 1] if "*" in p else c_type
            assert _c_type_matches(c_type, ct), (name, p, ct)
        assert _c_type_matches(ret.strip(), res), (name, ret, res)


def test_status_strings(lib):
    assert avtp.status_string(avtp.OK) == "ok"
    assert "workspace" in avtp.status_string(avtp.ERR_WORKSPACE)
    assert avtp.status_string(12345) == "unknown status"
    assert lib.avtp_version() >= 100


def test_kept_count_matches_oracle_budget_rule(lib):
    rng = np.random.default_rng(17)
    for _ in range(50):
        R = int(rng.integers(1, 6))
        reqs = []
        for _ in range(R):
            segs = [("t", int(rng.integers(0, 50)))]
            for _ in range(int(rng.integers(0, 10))):
                segs += [("i", int(rng.integers(1, 2000))), ("t", int(rng.integers(0, 4)))]
            reqs.append(segs)
        lay = synth.Layout.from_segments(reqs)
        kr = rng.choice(np.array([0.0, 0.05, 0.125, 0.25, 0.33, 0.5, 0.7, 1.0], dtype=np.float32), size=R)
        host = dict(cu_seqlens=lay.cu_seqlens, img_cu=lay.img_cu, img_len=lay.img_len)
        expect = 0
        vis = lay.n_visual_per_request()
        for r in range(R):
            T_r = int(lay.cu_seqlens[r + 1] - lay.cu_seqlens[r])
            expect += O.global_budget(kr[r], int(vis[r])) + T_r - int(vis[r])
        assert avtp.kept_count_host(host, kr) == expect


def test_kept_count_from_visual_counts_matches_the_layout_form(lib):
    # avtp_kept_count_vis_host sizes a later progressive stage from per-request visual
    # counts; its total, offsets and kept visual counts follow the oracle's budget rule
    rng = np.random.default_rng(23)
    for _ in range(50):
        R = int(rng.integers(1, 6))
        reqs = []
        for _ in range(R):
            segs = [("t", int(rng.integers(0, 40)))]
            for _ in range(int(rng.integers(0, 8))):
                segs += [("i", int(rng.integers(1, 1500))), ("t", int(rng.integers(0, 4)))]
            reqs.append(segs)
        lay = synth.Layout.from_segments(reqs)
        kr = rng.choice(np.array([0.0, 0.05, 0.25, 0.33, 0.5, 0.79, 1.0], dtype=np.float32), size=R)
        vis = lay.n_visual_per_request().astype(np.int32)
        n, out_cu, out_nv = avtp.kept_count_vis_host(lay.cu_seqlens, vis, kr)
        host = dict(cu_seqlens=lay.cu_seqlens, img_cu=lay.img_cu, img_len=lay.img_len)
        assert n == avtp.kept_count_host(host, kr)
        assert out_cu[0] == 0 and out_cu[-1] == n
        for r in range(R):
            kept_vis = O.global_budget(kr[r], int(vis[r]))
            assert out_nv[r] == kept_vis
            T_r = int(lay.cu_seqlens[r + 1] - lay.cu_seqlens[r])
            assert out_cu[r + 1] - out_cu[r] == kept_vis + T_r - int(vis[r])
    with pytest.raises(avtp.AVTPError):  # more visual tokens than the request holds
        avtp.kept_count_vis_host(np.array([0, 4], dtype=np.int32), np.array([5], dtype=np.int32),
                                 np.array([0.5], dtype=np.float32))


def test_kept_count_rejects_bad_ratio(lib):
    host = dict(cu_seqlens=np.array([0, 10]), img_cu=np.array([0, 1]), img_len=np.array([5]))
    with pytest.raises(avtp.AVTPError):
        avtp.kept_count_host(host, np.array([1.5], dtype=np.float32))


FAKE = 0x7f0000000000  # a 256-aligned address that is never dereferenced on these paths


def _layout(n_req=1, n_img=1, T=100):
    return avtp._Layout(n_req, n_img, T, FAKE, FAKE, FAKE, FAKE)


def _hv_args(hidden=64):
    a = avtp._ScoreArgs()
    a.criterion = avtp.CRIT_HIDDEN_VARIATION
    a.h_cur = a.h_prior = FAKE
    a.hidden, a.h_cur_stride, a.h_prior_stride = hidden, hidden, hidden
    return a


def _attn_args(d=128, hq=32, hkv=8):
    a = avtp._ScoreArgs()
    a.criterion = avtp.CRIT_TEXT_ATTENTION
    a.q = a.k = FAKE
    a.n_q_heads, a.n_kv_heads, a.head_dim = hq, hkv, d
    a.q_stride, a.k_stride = hq * d, hkv * d
    a.softmax_scale = d ** -0.5
    return a


def _score(lib, lay, args, ws_bytes=1 << 30, ws=FAKE):
    return lib.avtp_score(ctypes.byref(lay), ctypes.byref(args), FAKE, FAKE, ws, ws_bytes, None)


def test_host_validation_of_score_arguments(lib):
    assert lib.avtp_score(None, ctypes.byref(_hv_args()), FAKE, FAKE, FAKE, 1 << 30, None) == avtp.ERR_INVALID_ARG
    assert _score(lib, _layout(n_req=0), _hv_args()) == avtp.ERR_INVALID_ARG
    assert _score(lib, _layout(T=-1), _hv_args()) == avtp.ERR_INVALID_ARG
    assert _score(lib, _layout(T=1 << 31), _hv_args()) == avtp.ERR_RANGE
    assert _score(lib, _layout(), _hv_args(hidden=60)) == avtp.ERR_UNSUPPORTED
    assert _score(lib, _layout(), _attn_args(d=96)) == avtp.ERR_UNSUPPORTED
    assert _score(lib, _layout(), _attn_args(hq=30, hkv=8)) == avtp.ERR_UNSUPPORTED
    assert _score(lib, _layout(), _attn_args(hq=256, hkv=1)) == avtp.ERR_UNSUPPORTED  # more than 128 heads per KV group
    bad = _attn_args()
    bad.softmax_scale = float("nan")
    assert _score(lib, _layout(), bad) == avtp.ERR_INVALID_ARG
    misaligned = _hv_args()
    misaligned.h_cur = FAKE + 8
    assert _score(lib, _layout(), misaligned) == avtp.ERR_UNSUPPORTED
    assert _score(lib, _layout(), _hv_args(), ws_bytes=512) == avtp.ERR_WORKSPACE
    assert _score(lib, _layout(), _hv_args(), ws=FAKE + 16) == avtp.ERR_WORKSPACE
    crit = _hv_args()
    crit.criterion = 7
    assert _score(lib, _layout(), crit) == avtp.ERR_INVALID_ARG


def test_host_validation_of_alloc_and_compact_arguments(lib):
    lay = _layout()
    for alpha, r_min, r_max in [(float("nan"), 0.05, 0.95), (-1.0, 0.05, 0.95), (2048.0, 0.05, 0.95),
                                (1.0, 0.5, 0.4), (1.0, -0.1, 0.9), (1.0, 0.1, 1.5)]:
        aa = avtp._AllocArgs(FAKE, alpha, r_min, r_max, 0)
        assert lib.avtp_allocate(ctypes.byref(lay), FAKE, ctypes.byref(aa), FAKE, FAKE, FAKE, 1 << 30,
                                 None) == avtp.ERR_INVALID_ARG
    rows = (avtp._Rows * 9)()
    for i in range(9):
        rows[i] = avtp._Rows(FAKE, FAKE, 16, 16, 16)
    assert lib.avtp_compact(FAKE, 10, 100, rows, 9, FAKE, 1 << 20, None) == avtp.ERR_INVALID_ARG
    rows[0] = avtp._Rows(FAKE, FAKE, 32, 16, 32)  # stride shorter than the row
    assert lib.avtp_compact(FAKE, 10, 100, rows, 1, FAKE, 1 << 20, None) == avtp.ERR_INVALID_ARG
    rows[0] = avtp._Rows(FAKE, FAKE, 16, 16, 16)
    assert lib.avtp_compact(FAKE, 10, 100, rows, 1, None, 1 << 20, None) == avtp.ERR_WORKSPACE
    assert lib.avtp_compact(FAKE, -1, 100, rows, 1, FAKE, 1 << 20, None) == avtp.ERR_INVALID_ARG
    rows[0] = avtp._Rows(None, FAKE, 16, 16, 16)  # a NULL row pointer with rows to gather
    assert lib.avtp_compact(FAKE, 10, 100, rows, 1, FAKE, 1 << 20, None) == avtp.ERR_INVALID_ARG
    rows[0] = avtp._Rows(FAKE, None, 16, 16, 16)
    assert lib.avtp_compact(FAKE, 10, 100, rows, 1, FAKE, 1 << 20, None) == avtp.ERR_INVALID_ARG


def test_workspace_size_grows_with_attention_bookkeeping(lib):
    lay = _layout(n_req=2, n_img=5, T=10000)
    a = ctypes.c_size_t()
    b = ctypes.c_size_t()
    assert lib.avtp_workspace_size(ctypes.byref(lay), ctypes.byref(_hv_args()), ctypes.byref(a)) == avtp.OK
    assert lib.avtp_workspace_size(ctypes.byref(lay), ctypes.byref(_attn_args()), ctypes.byref(b)) == avtp.OK
    assert b.value > a.value >= 10000 * 4
    assert a.value % 256 == 0 and b.value % 256 == 0


def _fwd_args(d=128, hq=32, hkv=8, T=100):
    return avtp._ForwardArgs(FAKE, hkv * d, FAKE, hq * d, FAKE, T)


def _forward(lib, lay, sa, fa, scores=FAKE, sums=FAKE, ws=FAKE, ws_bytes=1 << 34):
    return lib.avtp_attn_forward(ctypes.byref(lay), ctypes.byref(sa) if sa is not None else None,
                                 ctypes.byref(fa) if fa is not None else None, scores, sums, ws, ws_bytes, None)


def test_host_validation_of_forward_arguments(lib):
    lay = _layout(T=100)
    assert _forward(lib, lay, None, _fwd_args()) == avtp.ERR_INVALID_ARG
    assert _forward(lib, lay, _attn_args(), None) == avtp.ERR_INVALID_ARG
    assert _forward(lib, lay, _hv_args(), _fwd_args()) == avtp.ERR_INVALID_ARG  # the criterion of the forward is B
    supplied = _attn_args()
    supplied.lse, supplied.lse_stride = FAKE, 100  # the forward writes the LSE itself
    assert _forward(lib, lay, supplied, _fwd_args()) == avtp.ERR_INVALID_ARG
    assert _forward(lib, lay, _attn_args(d=96), _fwd_args(d=96)) == avtp.ERR_UNSUPPORTED
    for field, value, code in [("v", None, avtp.ERR_INVALID_ARG), ("o", None, avtp.ERR_INVALID_ARG),
                               ("lse", None, avtp.ERR_INVALID_ARG), ("v", FAKE + 8, avtp.ERR_UNSUPPORTED),
                               ("o", FAKE + 4, avtp.ERR_UNSUPPORTED), ("v_stride", 8 * 128 - 8, avtp.ERR_INVALID_ARG),
                               ("v_stride", 8 * 128 + 4, avtp.ERR_UNSUPPORTED),
                               ("o_stride", 32 * 128 + 2, avtp.ERR_UNSUPPORTED),
                               ("o_stride", 32 * 128 - 4, avtp.ERR_INVALID_ARG),
                               ("lse_stride", 99, avtp.ERR_INVALID_ARG)]:
        fa = _fwd_args()
        setattr(fa, field, value)
        assert _forward(lib, lay, _attn_args(), fa) == code, (field, value)
    assert _forward(lib, lay, _attn_args(), _fwd_args(), sums=None) == avtp.ERR_INVALID_ARG  # both or neither
    assert _forward(lib, lay, _attn_args(), _fwd_args(), ws_bytes=1024) == avtp.ERR_WORKSPACE
    assert _forward(lib, lay, _attn_args(), _fwd_args(), ws=FAKE + 16) == avtp.ERR_WORKSPACE


def test_forward_workspace_holds_the_transposed_values(lib):
    lay = _layout(n_req=2, n_img=5, T=10000)
    a, b = ctypes.c_size_t(), ctypes.c_size_t()
    sa = _attn_args()
    assert lib.avtp_workspace_size(ctypes.byref(lay), ctypes.byref(sa), ctypes.byref(a)) == avtp.OK
    fa = _fwd_args(T=10000)
    assert lib.avtp_forward_workspace_size(ctypes.byref(lay), ctypes.byref(sa), ctypes.byref(fa),
                                           ctypes.byref(b)) == avtp.OK
    assert b.value >= 8 * 128 * 10000 * 2 and b.value % 256 == 0


def test_forward_timeline_needs_the_timeline_build(lib):
    out = np.zeros((4, 10), dtype=np.int64)
    assert lib.avtp_forward_timeline(out.ctypes.data, 4) == avtp.ERR_UNSUPPORTED
    assert lib.avtp_score_timeline(1, out.ctypes.data, 4) == avtp.ERR_UNSUPPORTED


def test_host_validation_of_wait_selftest_arguments(lib):
    for bad in (-1, 0, 999, 10_000_000_001):
        assert lib.avtp_wait_selftest(bad, 0, FAKE, 256, None) == avtp.ERR_INVALID_ARG
    assert lib.avtp_wait_selftest(1_000_000, 0, None, 256, None) == avtp.ERR_WORKSPACE
    assert lib.avtp_wait_selftest(1_000_000, 0, FAKE + 8, 256, None) == avtp.ERR_WORKSPACE
    assert lib.avtp_wait_selftest(1_000_000, 0, FAKE, 8, None) == avtp.ERR_WORKSPACE


def test_binding_structs_match_the_c_layout(tmp_path):
    if shutil.which("gcc") is None:
        pytest.skip("needs a host C compiler")
    # sizeof and every field offset of the ABI structs, from the header compiled by the
    # host C compiler, against the ctypes mirrors of the binding
    structs = {"avtp_layout_t": avtp._Layout, "avtp_score_args_t": avtp._ScoreArgs,
               "avtp_alloc_args_t": avtp._AllocArgs, "avtp_rows_t": avtp._Rows,
               "avtp_forward_args_t": avtp._ForwardArgs}
    renamed = {"in_": "in"}  # a Python keyword in the mirror
    lines = ["#include <stdio.h>", "#include <stddef.h>", '#include "avtp.h"', "int main(void) {"]
    for c_name, py in structs.items():
        lines.append(f'  printf("{c_name} size %zu\\n", sizeof({c_name}));')
        for f, _ in py._fields_:
            cf = renamed.get(f, f)
            lines.append(f'  printf("{c_name} {f} %zu\\n", offsetof({c_name}, {cf}));')
    lines += ["  return 0;", "}"]
    src = tmp_path / "abi.c"
    src.write_text("\n".join(lines) + "\n")
    exe = tmp_path / "abi"
    cc = subprocess.run(["gcc", "-std=c11", "-I", os.path.dirname(HEADER), str(src), "-o", str(exe)],
                        capture_output=True, text=True)
    assert cc.returncode == 0, cc.stderr
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split("\n")
    got = {}
    for ln in out:
        if ln:
            c_name, field, value = ln.split()
            got[(c_name, field)] = int(value)
    for c_name, py in structs.items():
        assert got[(c_name, "size")] == ctypes.sizeof(py), c_name
        for f, _ in py._fields_:
            assert got[(c_name, f)] == getattr(py, f).offset, (c_name, f)

