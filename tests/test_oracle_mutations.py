"""Plant plausible mistakes in a copy of the oracle and check that a pin catches each.

Each mutation edits the oracle's source text (a dropped term, a flipped sign, a
wrong index, a transposed operand, a wrong mean), loads it as a fresh module and
runs the pin tests of ``test_oracle_pins`` against it. At least one pin must
fail. CPU only; the real oracle is untouched.
"""
import importlib.util
import inspect
import os
import sys
import types

import pytest

import tests.test_oracle_pins as pins
from oracle import avtp_oracle

SRC_PATH = inspect.getsourcefile(avtp_oracle)

MUTATIONS = {
    "ratio sign flipped": ("return [r_base + alpha * (ib - avg) for ib in ibar]",
                           "return [r_base - alpha * (ib - avg) for ib in ibar]"),
    "ratio off by a factor of two": ("return [Fraction(int(S[i]), (1 << FX_FRAC_BITS) * int(n[i])) for i in range(len(n))]",
                                     "return [Fraction(int(S[i]), (1 << (FX_FRAC_BITS - 1)) * int(n[i])) for i in range(len(n))]"),
    "image-weighted mean": ("return Fraction(sum(int(v) for v in S), (1 << FX_FRAC_BITS) * sum(int(v) for v in n))",
                            "return sum(image_means(S, n), Fraction(0)) / len(n)"),
    "relative rule drops r_base": ("return [r_base * (1 + alpha * (ib / avg - 1)) for ib in ibar]",
                                   "return [(1 + alpha * (ib / avg - 1)) for ib in ibar]"),
    "relative rule ignores alpha": ("return [r_base * (1 + alpha * (ib / avg - 1)) for ib in ibar]",
                                    "return [r_base * (ib / avg) for ib in ibar]"),
    "GQA head mapping": ("g = h // (n_q_heads // n_kv_heads)", "g = h % n_kv_heads"),
    "causal mask off by one": ("visible = keys[None, :] <= qpos[:, None]",
                               "visible = keys[None, :] < qpos[:, None]"),
    "logits transposed": ("z = float(scale) * (Qh @ Kg.T)",
                          "z = float(scale) * (Kg @ Qh.T).T[:, ::-1]"),
    "norm of wrong row": ("nb = np.sqrt(np.sum(b * b, axis=1))", "nb = np.sqrt(np.sum(a * a, axis=1))"),
    "cosine not subtracted": ("out[rows] = 1.0 - cos", "out[rows] = cos"),
    "query count dropped": ("out[a:b][vis] = acc[vis] / (n_q_heads * nq)", "out[a:b][vis] = acc[vis] / n_q_heads"),
    "remainder tie to higher index": ("order = sorted(elig, key=lambda i: (-frac[i], i))",
                                      "order = sorted(elig, key=lambda i: (-frac[i], -i))"),
    "no clamp": ("return min(max(x, lo), hi)", "return x"),
    "water-fill takes the last short breakpoint": ("return pts[k] + (B - G[k]) * (pts[k + 1] - pts[k]) / (G[k + 1] - G[k])",
                                                   "return pts[k]"),
    "remainder from the wrong end": ("frac = [v - math.floor(v) for v in x]", "frac = [1 - (v - math.floor(v)) for v in x]"),
    "budget rounding floor": ("return math.floor(Fraction(float(np.float32(keep_ratio_f32))) * int(n_vis) + Fraction(1, 2))",
                              "return math.floor(Fraction(float(np.float32(keep_ratio_f32))) * int(n_vis))"),
    "ties by higher position": ("return (0, -score, pos)", "return (0, -score, -pos)"),
    "NaN ranked high": ("return (1, 0.0, pos)", "return (-1, 0.0, pos)"),
    "text dropped": ("keep = ~_request_visual_local(layout, r)  # text always kept",
                     "keep = np.zeros(b - a, dtype=bool)"),
    "fixed point truncates": ("return np.rint(s * float(2 ** FX_FRAC_BITS)).astype(np.int64)",
                              "return np.trunc(s * float(2 ** FX_FRAC_BITS)).astype(np.int64)"),
    "last query set takes the first token": ("return np.arange(T_r - 1, T_r) if T_r > 0 else np.zeros(0, dtype=np.int64)",
                                             "return np.arange(0, 1) if T_r > 0 else np.zeros(0, dtype=np.int64)"),
    "layers ranked in ascending attention": ("order = sorted(range(L), key=lambda l: (-int(A[i, l]), l))",
                                             "order = sorted(range(L), key=lambda l: (int(A[i, l]), l))"),
    "layer ties to the higher index": ("order = sorted(range(L), key=lambda l: (-int(A[i, l]), l))",
                                       "order = sorted(range(L), key=lambda l: (-int(A[i, l]), -l))"),
    "layers chosen by the worst mean rank": ("order = sorted(range(len(rank_sum)), key=lambda l: (int(rank_sum[l]), l))",
                                             "order = sorted(range(len(rank_sum)), key=lambda l: (-int(rank_sum[l]), l))"),
    "layer mass misses the last image": ("out[r] = sum(int(v) for v in img_sums[int(layout.img_cu[r]):int(layout.img_cu[r + 1])])",
                                         "out[r] = sum(int(v) for v in img_sums[int(layout.img_cu[r]):int(layout.img_cu[r + 1]) - 1])"),
    "pruned image starts after its first kept token": ("starts.append(int(np.count_nonzero(local < s0)))",
                                                       "starts.append(int(np.count_nonzero(local <= s0)))"),
    "forward takes values from the wrong KV head": ("O[a + qpos, h, :] = P @ bf16_to_f64(v[a:b, h // G, :])",
                                                    "O[a + qpos, h, :] = P @ bf16_to_f64(v[a:b, h % n_kv_heads, :])"),
    "forward normaliser in base 2": ("lse[h, a + qpos] = norm", "lse[h, a + qpos] = norm / np.log(2.0)"),
    "forward query set skips the first token": ("        return np.arange(T_r)\n", "        return np.arange(1, T_r)\n"),
    "forward rows see the next key": ("Kg = bf16_to_f64(k[a:a + p + 1, g, :])", "Kg = bf16_to_f64(k[a:a + p + 2, g, :])"),
    "forward rows weight values unnormalised": ("O[j, h, :] = (w / np.sum(w)) @ bf16_to_f64(v[a:a + p + 1, g, :])",
                                                "O[j, h, :] = w @ bf16_to_f64(v[a:a + p + 1, g, :])"),
    "pruned image span keeps its old length": ("lens.append(int(np.count_nonzero((local >= s0) & (local < s1))))",
                                               "lens.append(s1 - s0)"),
}

PIN_TESTS = [name for name, fn in inspect.getmembers(pins, inspect.isfunction) if name.startswith("test_")]


def _mutant(old, new):
    src = open(SRC_PATH).read()
    assert src.count(old) == 1, f"mutation anchor not found exactly once: {old!r}"
    mod = types.ModuleType("avtp_oracle_mutant")
    exec(compile(src.replace(old, new), "avtp_oracle_mutant", "exec"), mod.__dict__)
    return mod


def _run_pins(module, monkeypatch):
    monkeypatch.setattr(pins, "O", module)
    failures = []
    for name in PIN_TESTS:
        fn = getattr(pins, name)
        params = getattr(fn, "pytestmark", [])
        arg_sets = [()]
        for mark in params:
            if mark.name == "parametrize":
                arg_sets = [v if isinstance(v, tuple) else (v,) for v in mark.args[1]]
        for args in arg_sets:
            try:
                fn(*args)
            except Exception:  # noqa: BLE001 - any failure counts as caught
                failures.append(name)
                break
    return failures


def test_unmutated_oracle_passes_every_pin(monkeypatch):
    assert _run_pins(avtp_oracle, monkeypatch) == []


# a mutant may compute with inf or NaN (for example a mask that lets -inf through)
@pytest.mark.filterwarnings("ignore::RuntimeWarning")
@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_mutation_is_caught(name, monkeypatch):
    old, new = MUTATIONS[name]
    failures = _run_pins(_mutant(old, new), monkeypatch)
    assert failures, f"no pin caught the planted mistake: {name}"
