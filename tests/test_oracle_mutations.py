"""Mutation check of the oracle pins: plausible mistakes are planted in a copy of
the oracle's source (on the CPU, never in the CUDA path) and each must make at
least one pin of tests/test_oracle_pins.py fail."""

import inspect
import sys
import types

import pytest

import tests.test_oracle_pins as pins
from oracle import kashin_oracle as ko

SRC = inspect.getsource(ko)

MUTANTS = {
    "dct_no_row0_scale": ("C[0, :] *= 1.0 / np.sqrt(2.0)", "C[0, :] *= 1.0"),
    "dct_wrong_phase": ("(2.0 * n + 1.0) * j", "(2.0 * n) * j"),
    "divisor_N_minus_1": ("lam = np.abs(rho).sum(axis=0) / N", "lam = np.abs(rho).sum(axis=0) / (N - 1)"),
    "v_divisor_N_minus_1": ("lam = np.abs(y).sum(axis=0) / N", "lam = np.abs(y).sum(axis=0) / (N - 1)"),
    "u_update_sign": ("rho = rho - du", "rho = rho + du"),
    "v_update_without_P": ("rho = rho - P(dv)", "rho = rho - dv"),
    "sign_zero_is_plus": ("return np.sign(a)", "return np.where(a >= 0, 1.0, -1.0)"),
    "no_sign_flip": ("a = self.eps[:, None] * a", "a = a"),
    "centre_inner_no_abs": ("inner = np.abs(a1 - a2)", "inner = a1 - a2"),
    "codes_tie_upper": ("out += (v32 > b[None, :, i])", "out += (v32 >= b[None, :, i])"),
    "pack_shift": ("<< np.uint64(2 * (i % 16))", "<< np.uint64(2 * (15 - i % 16))"),
    "mask_low_bit": ("out[j] = -1.0 if (z >> 63) else 1.0", "out[j] = -1.0 if (z & 1) else 1.0"),
    "kmeans_empty_to_zero": ("c[:, q] = np.where(cnt > 0, tot / np.maximum(cnt, 1), c[:, q])",
                             "c[:, q] = tot / np.maximum(cnt, 1)"),
    "kmeans_sum_not_mean": ("c[:, q] = np.where(cnt > 0, tot / np.maximum(cnt, 1), c[:, q])",
                            "c[:, q] = np.where(cnt > 0, tot, c[:, q])"),
    "alg2_literal_projection": ("c = float(y @ s) / nnz if nnz else 0.0", "c = float(r @ s) / nnz if nnz else 0.0"),
    "alg2_branch_reversed": ("if np.abs(r).sum() > np.abs(y).sum():", "if np.abs(r).sum() < np.abs(y).sum():"),
    "alg2_v_update_without_Q": ("r = r - Q(c * s)", "r = r - c * s"),
    "rht_no_normalisation": ("Hn = hadamard_matrix(b) / np.sqrt(b)", "Hn = hadamard_matrix(b)"),
    "rht_signs_after_transform": ("z = x if inverse else s * x\n    y = np.empty_like(z)\n"
                                  "    for k in range(n // b):\n"
                                  "        y[k * b:(k + 1) * b] = Hn @ z[k * b:(k + 1) * b]\n"
                                  "    if inverse:\n        y = s * y",
                                  "z = x\n    y = np.empty_like(z)\n"
                                  "    for k in range(n // b):\n"
                                  "        y[k * b:(k + 1) * b] = Hn @ z[k * b:(k + 1) * b]\n"
                                  "    if True:\n        y = s * y"),
    "rht_whole_vector_block": ("    b = n & -n\n    return min(b, RHT_MAX_BLOCK)", "    return n"),
    "hadamard_wrong_sign_block": ("H = np.block([[H, H], [H, -H]])", "H = np.block([[H, H], [-H, H]])"),
    "reverse_schedule_u_second": ("for j in (1, 2):                     # two greedy steps from Q_N",
                                  "for j in ():"),
}


def _load_mutant(name):
    old, new = MUTANTS[name]
    assert SRC.count(old) >= 1, f"mutation anchor for {name} not found"
    src = SRC.replace(old, new)
    return _exec_module(f"ko_mutant_{name}", src)


def _exec_module(modname, src):
    mod = types.ModuleType(modname)
    sys.modules[modname] = mod          # dataclasses resolve annotations through sys.modules
    exec(compile(src, f"<{modname}>", "exec"), mod.__dict__)
    return mod


def _run_all_pins(mod, monkeypatch):
    monkeypatch.setattr(pins, "ko", mod)
    failures = 0
    for fname, fn in inspect.getmembers(pins, inspect.isfunction):
        if not fname.startswith("test_"):
            continue
        marks = getattr(fn, "pytestmark", [])
        cases = [()]
        for m in marks:
            if m.name == "parametrize":
                argnames = [a.strip() for a in m.args[0].split(",")]
                cases = [v if isinstance(v, tuple) else (v,) for v in m.args[1]]
                cases = [dict(zip(argnames, c)) for c in cases]
        for c in cases:
            try:
                if isinstance(c, dict):
                    fn(**c)
                else:
                    fn()
            except (AssertionError, Exception):
                failures += 1
    return failures


@pytest.mark.parametrize("name", sorted(MUTANTS))
def test_mutant_is_caught(name, monkeypatch):
    mod = _load_mutant(name)
    assert _run_all_pins(mod, monkeypatch) > 0, f"mutation {name} survived every pin"


def test_unmutated_oracle_passes_all(monkeypatch):
    mod = _exec_module("ko_copy", SRC)
    assert _run_all_pins(mod, monkeypatch) == 0
