"""GPU parity tests of the run-time-length path: the vector lengths without a
compiled plan (any 1 <= n <= 16384 whose prime factors lie in {2, 3, 5, 7, 11, 13,
43}), through the same C ABI calls, against the fp64 oracle.

Lengths cover every radix of the path (16, 8, 4, 2, 9, 3, 5, 7, 11, 13, 43), odd n
(Makhoul's reordering with ceil(n/2) even positions), n < 16 (a single, partly
filled code word), the self-paired frequencies 0 and n/2, and model widths
without a tuned plan (2560, 5120, 6144, 13824)."""

import numpy as np
import pytest

from oracle import kashin_oracle as ko
from tests import parity

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def kd():
    import torch
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2609_11687_gb300 import build
    build.build()
    from paper_2609_11687_gb300 import kashin
    return kashin


@pytest.fixture(scope="module")
def torch_mod():
    import torch
    return torch


def _rand(torch, shape, seed, dtype=None, scale=0.02):
    g = torch.Generator().manual_seed(seed)
    x = torch.randn(shape, generator=g) * scale
    return x if dtype is None else x.to(dtype)


APPLY_N = [1, 2, 3, 5, 6, 7, 9, 10, 11, 12, 13, 15, 43, 86, 100, 105, 129, 640, 1000, 2560, 4095, 5120, 6144,
           13824]


def test_lengths_are_generic(kd):
    for n in APPLY_N:
        assert kd.kd_supported(n) == kd.KD_OK and not kd.kd_tuned(n), n


@pytest.mark.parametrize("n", APPLY_N)
def test_generic_apply_p_matches_dense(kd, torch_mod, n):
    torch = torch_mod
    m = 7  # odd: the last pair has one vector
    x = _rand(torch, (m, n), seed=n, scale=1.0)
    y = kd.apply_p(x.cuda(), sign_seed=n + 5).cpu().numpy().astype(np.float64)
    P = ko.POperator(n, ko.sign_mask(n + 5, n))
    ref = P(x.numpy().astype(np.float64).T).T
    rms = np.sqrt((x.numpy().astype(np.float64) ** 2).mean(axis=1, keepdims=True))
    err = np.abs(y - ref) / rms
    assert err.max() < 1e-5, err.max()
    l2 = np.linalg.norm(y - ref, axis=1) / np.linalg.norm(ref, axis=1)
    assert l2.max() < 2e-6, l2.max()


@pytest.mark.parametrize("n", [2, 100, 1000, 5120])
def test_generic_apply_p_is_involution(kd, torch_mod, n):
    torch = torch_mod
    x = _rand(torch, (4, n), seed=3, scale=1.0).cuda()
    y = kd.apply_p(kd.apply_p(x, 9), 9)
    assert (y - x).abs().max().item() < 2e-5


def _parity(kd, torch, G_cpu, seed, iters=16, layout="rows", kmeans_iters=0):
    w = G_cpu.cuda()
    if layout == "columns":
        w = G_cpu.t().contiguous().cuda()
    dev = parity.device_outputs(kd, w, iters, seed, trace=True, layout=layout, kmeans_iters=kmeans_iters)
    x = G_cpu.to(torch.float64).numpy().T
    return parity.compare(x, seed, iters, dev, kmeans_iters=kmeans_iters), dev


@pytest.mark.parametrize("n,m", [(1, 3), (2, 5), (3, 5), (10, 5), (43, 5), (100, 7), (105, 5), (640, 9),
                                 (1000, 5), (2560, 5), (5120, 3), (13824, 3)])
def test_generic_parity(kd, torch_mod, n, m):
    torch = torch_mod
    G = _rand(torch, (m, n), seed=n + 17)
    rep, _ = _parity(kd, torch, G, seed=n + 1)
    print(rep)
    # n = 2: the second step zeroes the residual (both entries have the same
    # magnitude after the first), so vhat = 0 and all its boundaries are 0: every
    # vhat entry sits on a boundary by construction, as for a constant vector
    rep.check(code_budget=n > 2)


def test_generic_fp16_columns_and_kmeans(kd, torch_mod):
    torch = torch_mod
    G = _rand(torch, (6, 2560), seed=41, dtype=torch.float16)
    rep, _ = _parity(kd, torch, G, seed=43, layout="columns", kmeans_iters=3)
    rep.check()


@pytest.mark.parametrize("iters", [0, 1, 3])
def test_generic_iteration_counts(kd, torch_mod, iters):
    torch = torch_mod
    G = _rand(torch, (5, 100), seed=iters + 50)
    rep, dev = _parity(kd, torch, G, 77, iters=iters)
    rep.check()
    if iters == 0:
        assert not dev["u"].any() and not dev["vhat"].any()
        np.testing.assert_array_equal(dev["resid"], G.numpy())
        assert not dev["words_u"].any() and not dev["words_v"].any()


def test_generic_degenerate_vectors(kd, torch_mod):
    torch = torch_mod
    G = _rand(torch, (6, 100), seed=4)
    G[1] = 0.0                           # all-zero vector
    G[2, ::3] = 0.0                      # exact zeros
    G[3, :] = 0.0
    G[3, 17] = 0.5                       # a single spike
    G[4] = 1e-3                          # constant vector
    rep, dev = _parity(kd, torch, G, seed=5, kmeans_iters=2)
    rep.check(code_budget=False)
    assert not dev["u"][1].any() and not dev["vhat"][1].any()
    assert not dev["centres_u"][1].any() and not dev["words_u"][1].any()


def test_generic_tail_word_is_zero_padded(kd, torch_mod):
    """n = 100: seven code words per vector; entries 100..111 of the last word are 0."""
    torch = torch_mod
    G = _rand(torch, (4, 100), seed=9)
    d = kd.decompose(G.cuda(), 8, 3)
    torch.cuda.synchronize()
    assert tuple(d.codes_u.shape) == (4, 7)
    for words in (d.codes_u, d.codes_v):
        last = words[:, 6].cpu().numpy().astype(np.uint32)
        assert not (last >> np.uint32(8)).any()   # bits of entries 100..111


def test_generic_trace_and_factors_do_not_change_results(kd, torch_mod):
    torch = torch_mod
    w = _rand(torch, (9, 5120), seed=8, dtype=torch.float16).cuda()
    a = kd.decompose(w, 16, 3, factors=True, trace=True)
    b = kd.decompose(w, 16, 3, factors=False, coeffs=False, trace=False)
    torch.cuda.synchronize()
    for name in ("codes_u", "codes_v", "centres_u", "centres_v"):
        assert torch.equal(getattr(a, name), getattr(b, name)), name


def test_generic_batch_equals_single(kd, torch_mod):
    """kd_decompose_batch runs the run-time-length path one matrix at a time."""
    torch = torch_mod
    ws = [_rand(torch, (5, 640), seed=60).cuda(), _rand(torch, (2, 640), seed=61).cuda()]
    assert not kd.kd_batchable(640)
    bat = kd.decompose_batch(ws, 8, [3, 4])
    for w, sd, b in zip(ws, [3, 4], bat):
        one = kd.decompose(w, 8, sd)
        torch.cuda.synchronize()
        for name in ("codes_u", "codes_v", "centres_u", "centres_v"):
            assert torch.equal(getattr(one, name), getattr(b, name)), name


@pytest.mark.parametrize("n,m", [(100, 5), (2560, 4)])
def test_generic_reconstruct_matches_oracle(kd, torch_mod, n, m):
    torch = torch_mod
    G = _rand(torch, (m, n), seed=n + 3)
    d = kd.decompose(G.cuda(), 16, 21, kmeans_iters=2)
    W_hat = kd.reconstruct(d, n, 21)
    W_cols = kd.reconstruct(d, n, 21, layout="columns", dtype=torch.float16)
    torch.cuda.synchronize()
    ref = ko.reconstruct(kd.unpack_codes(d.codes_u, n).T, kd.unpack_codes(d.codes_v, n).T,
                         d.centres_u.double().cpu().numpy(), d.centres_v.double().cpu().numpy(),
                         ko.sign_mask(21, n)).T                             # (m, n)
    scale = np.abs(ref).max()
    assert np.abs(W_hat.double().cpu().numpy() - ref).max() <= 1e-5 * scale
    assert torch.equal(W_cols.t(), W_hat.half())
