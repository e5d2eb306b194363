"""The bench's fixed conventions, checked on the host: the algorithmic flop count
of one vector (four length-n DCTs per block at 2 n log2 n plus 20 n for the four
greedy steps) against its per-parameter values at k = 16, the algorithmic bytes of
the n = 4096 launch, and the profile hash ignoring comment-only edits."""

import importlib.util
import math
import os

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def bench():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


# per-parameter flops at k = 16 as tabulated (to the nearest unit or truncated):
# k (8 log2 n + 20)
PER_PARAM_K16 = {256: 1344, 768: 1547, 3072: 1803, 4096: 1856, 11008: 2038, 14336: 2087, 16384: 2112}


@pytest.mark.parametrize("n,expect", sorted(PER_PARAM_K16.items()))
def test_flop_convention_per_parameter(bench, n, expect):
    assert abs(bench.flops_per_vector(n, 16) / n - expect) < 1.0
    # linear in the block count, zero at k = 0
    assert bench.flops_per_vector(n, 0) == 0
    assert math.isclose(bench.flops_per_vector(n, 32), 2 * bench.flops_per_vector(n, 16))


def test_fft_count_is_the_conventional_secondary(bench):
    # 2.5 n log2 n per transform instead of 2 n log2 n: strictly above the primary count
    for n in PER_PARAM_K16:
        assert bench.fft_flops_per_vector(n, 16) > bench.flops_per_vector(n, 16)


def test_profile_hash_ignores_comments(bench, tmp_path):
    src = "int f() { return 1; }  // one\n/* block\n comment */ int g();\n"
    same = "int f() {\n  return 1;  // other words\n}\nint g();\n"
    other = "int f() { return 2; }\nint g();\n"
    assert bench._code_only(src) == bench._code_only(same)
    assert bench._code_only(src) != bench._code_only(other)


def test_reference_arm_line_on_cpu():
    """The reference arm (the CPU oracle) runs without a GPU: one JSON line with
    impl = reference, the arm's own step time (each step one pass over the fixed
    sample), and cpu_baseline / e2e describing the same run."""
    import json
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    out = subprocess.run([sys.executable, os.path.join(root, "bench.py"), "--impl", "reference", "--workload", "w256",
                          "--steps", "2", "--warmup", "3"], capture_output=True, text=True, timeout=600, cwd=root)
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [l for l in out.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["steps"] == 2 and d["warmup"] == 3
    assert d["value"] > 0 and d["ms_per_step"] > 0 and d["higher_is_better"] is True
    assert d["config"]["sample_params_per_step"] == 256 * 256       # the whole 256 x 256 matrix
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["value"] == d["value"]
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["value"] == d["value"]
