"""kd_decompose_batch: several matrices of one vector length in one launch must
give, matrix by matrix, exactly what kd_decompose gives (the per-pair arithmetic
is the same; only the assignment of pairs to CTAs changes)."""

import pytest

from paper_2609_11687_gb300 import synth

pytestmark = pytest.mark.gpu

ITERS = 16


@pytest.fixture(scope="module")
def kd():
    import torch
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2609_11687_gb300 import build
    build.build()
    from paper_2609_11687_gb300 import kashin
    return kashin


def _mats(n, ms, seed, dtype=None, layout="rows"):
    import dataclasses
    import torch
    out = []
    for i, m in enumerate(ms):
        spec = dataclasses.replace(synth.llama7b_layer(2)[0], N=n, M=m, seed=seed + i)
        w = synth.generate(spec, device="cuda")
        if dtype is not None:
            w = w.to(dtype)
        if layout == "columns":
            w = w.t().contiguous()
        out.append((spec, w))
    return out


def _check_equal(kd, mats, layout="rows", kmeans_iters=0):
    import torch
    ws = [w for _, w in mats]
    seeds = [s.sign_seed for s, _ in mats]
    batch = kd.decompose_batch(ws, ITERS, seeds, layout=layout, coeffs=True, kmeans_iters=kmeans_iters)
    singles = [kd.decompose(w, ITERS, sd, layout=layout, coeffs=True, kmeans_iters=kmeans_iters)
               for w, sd in zip(ws, seeds)]
    torch.cuda.synchronize()
    for b, s1 in zip(batch, singles):
        for f in ("codes_u", "codes_v", "centres_u", "centres_v", "coeffs"):
            assert torch.equal(getattr(b, f), getattr(s1, f)), f


@pytest.mark.parametrize("n,ms", [(4096, [4096, 37, 1, 11008, 6]), (768, [768, 768, 768, 768, 3072]),
                                  (3072, [768, 5]), (256, [1, 2, 3, 4, 5, 6, 7, 8] * 4)])
def test_batch_equals_single_calls(kd, n, ms):
    _check_equal(kd, _mats(n, ms, seed=100 + n))


def test_batch_long_vectors_run_per_matrix(kd):
    # n = 11008 has no batched kernel: the call runs one launch per matrix
    _check_equal(kd, _mats(11008, [5, 64, 2], seed=9))


def test_batch_layouts_dtypes_kmeans_and_empty(kd):
    import torch
    _check_equal(kd, _mats(1024, [7, 300, 2], seed=3, dtype=torch.bfloat16, layout="columns"), layout="columns")
    _check_equal(kd, _mats(512, [9, 64], seed=4), kmeans_iters=2)
    # an empty matrix among others
    mats = _mats(256, [5, 0, 6], seed=5)
    _check_equal(kd, mats)


def test_batch_limits(kd):
    import torch
    w = torch.zeros((2, 256), device="cuda")
    with pytest.raises(ValueError):
        kd.decompose_batch([w] * 33, ITERS, list(range(33)))
    with pytest.raises(ValueError):
        kd.decompose_batch([], ITERS, [])
