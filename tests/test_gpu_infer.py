"""Inference with the Kashin representation (App. C): dequantised factor planes,
the folding identity  X W_hat = X U_q + (X P) V_q = [X | XP][U_q; V_q]  and the
dense re-materialisation W_hat = U_q + P V_q, against the fp64 oracle.

Dequantisation copies centres, so it is bit-exact in fp32 (and equal to the
round-to-nearest conversion of those values in fp16 / bf16).  The two products
differ only by fp32 rounding: tolerance 1e-5 of max|Y|."""

import numpy as np
import pytest

from oracle import kashin_oracle as ko
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


def _layer(kd, n, m, seed):
    import dataclasses
    spec = dataclasses.replace(synth.llama7b_layer(1)[0], N=n, M=m, seed=seed)
    w = synth.generate(spec, device="cuda")
    return spec, w, kd.decompose(w, ITERS, spec.sign_seed, kmeans_iters=2)


@pytest.mark.parametrize("n,m", [(256, 7), (768, 33), (4096, 10), (11008, 3)])
def test_dequantise_matches_oracle(kd, n, m):
    import torch
    spec, w, dec = _layer(kd, n, m, 11 + n)
    for codes, cent in ((dec.codes_u, dec.centres_u), (dec.codes_v, dec.centres_v)):
        ref = ko.dequantise(kd.unpack_codes(codes, n).T, cent.cpu().numpy().astype(np.float64)).T   # (m, n)
        got = kd.dequantise(codes, cent, n)
        cols = kd.dequantise(codes, cent, n, layout="columns")
        half = kd.dequantise(codes, cent, n, dtype=torch.float16)
        bf = kd.dequantise(codes, cent, n, dtype=torch.bfloat16)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(got.cpu().numpy(), ref.astype(np.float32))
        assert torch.equal(cols.t(), got)
        assert torch.equal(half, got.half())
        assert torch.equal(bf, got.bfloat16())


def test_dequantise_ragged_length_and_strides(kd):
    """n not a multiple of 16 (tail word), ld > n, unaligned output start."""
    import torch
    n, m = 100, 5
    g = torch.Generator().manual_seed(1)
    codes = torch.randint(0, 2**31 - 1, (m, 7), generator=g, dtype=torch.int32).cuda()
    cent = torch.sort(torch.randn((m, 4), generator=g), dim=1).values.cuda()
    ref = ko.dequantise(kd.unpack_codes(codes, n).T, cent.cpu().numpy().astype(np.float64)).T.astype(np.float32)
    big = torch.full((m, 131), -7.0, device="cuda")
    out = big[:, 3:103]
    kd.dequantise(codes, cent, n, out=out)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(out.cpu().numpy(), ref)
    assert bool((big[:, :3] == -7.0).all()) and bool((big[:, 103:] == -7.0).all())


@pytest.mark.parametrize("n", [768, 4096, 11008])
def test_reconstruct_batch_equals_single_calls(kd, n):
    """One batched launch over matrices with their own seeds and vector counts (odd,
    one, none) writes every W_hat exactly as its own kd_reconstruct call; n = 11008
    takes the one-launch-per-matrix path."""
    import torch
    g = torch.Generator().manual_seed(n + 3)
    words = (n + 15) // 16
    ms = [7, 1, 0, 40] if n < 11008 else [3, 0, 2]
    seeds = [11 * i + n for i in range(len(ms))]
    decs = []
    for m in ms:
        cu = torch.sort(torch.randn((m, 4), generator=g), dim=1).values.cuda()
        cv = torch.sort(torch.randn((m, 4), generator=g), dim=1).values.cuda()
        decs.append(kd.Decomposed(
            codes_u=torch.randint(-2**31, 2**31 - 1, (m, words), generator=g, dtype=torch.int32).cuda(),
            codes_v=torch.randint(-2**31, 2**31 - 1, (m, words), generator=g, dtype=torch.int32).cuda(),
            centres_u=cu, centres_v=cv, coeffs=None, u=None, vhat=None, resid=None, trace=None))
    for dtype, layout in ((torch.float32, "rows"), (torch.float16, "rows"), (torch.float32, "columns")):
        got = kd.reconstruct_batch(decs, n, seeds, dtype=dtype, layout=layout)
        for d, sd, o in zip(decs, seeds, got):
            one = kd.reconstruct(d, n, sd, dtype=dtype, layout=layout)
            torch.cuda.synchronize()
            assert torch.equal(o, one), (n, dtype, layout)


@pytest.mark.parametrize("n", [100, 4096])
@pytest.mark.parametrize("layout", ["rows", "columns"])
def test_dequantise_batch_equals_single_calls(kd, n, layout):
    """One batched launch over planes of different vector counts (one of them empty,
    one written into a strided view) writes every plane exactly as its own call."""
    import torch
    g = torch.Generator().manual_seed(n)
    words = (n + 15) // 16
    ms = [5, 0, 300, 1, 64]
    planes = [(torch.randint(-2**31, 2**31 - 1, (m, words), generator=g, dtype=torch.int32).cuda(),
               torch.sort(torch.randn((m, 4), generator=g), dim=1).values.cuda()) for m in ms]
    for dtype in (torch.float32, torch.float16, torch.bfloat16):
        outs = []
        for (c, _), m in zip(planes, ms):
            shape = (m, n + 24) if layout == "rows" else (n, m + 24)
            outs.append(torch.full(shape, -3.0, dtype=dtype, device="cuda")[:, 8:(n if layout == "rows" else m) + 8])
        got = kd.dequantise_batch(planes, n, dtype=dtype, layout=layout, outs=outs)
        for (c, cent), o in zip(planes, got):
            one = kd.dequantise(c, cent, n, dtype=dtype, layout=layout)
            torch.cuda.synchronize()
            assert torch.equal(o, one)
            assert bool((o._base[:, :8] == -3.0).all()) and bool((o._base[:, -16:] == -3.0).all())


@pytest.mark.parametrize("n,m,t", [(768, 33, 5), (4096, 12, 8), (11008, 6, 3)])
def test_folding_identity(kd, n, m, t):
    """App. C: X W_hat computed three ways -- dense W_hat from kd_reconstruct, the
    folded [X | XP][U_q; V_q] with XP from kd_apply_p, and the fp64 oracle."""
    import torch
    spec, w, dec = _layer(kd, n, m, 5 + n)
    X = torch.randn((t, n), generator=torch.Generator().manual_seed(n), dtype=torch.float32).cuda()
    W_hat = kd.reconstruct(dec, n, spec.sign_seed)                       # (m, n): rows are vectors
    Uq = kd.dequantise(dec.codes_u, dec.centres_u, n)
    Vq = kd.dequantise(dec.codes_v, dec.centres_v, n)
    XP = kd.apply_p(X, spec.sign_seed)
    torch.cuda.synchronize()
    hp = torch.backends.cuda.matmul.allow_tf32
    torch.backends.cuda.matmul.allow_tf32 = False
    try:
        Y_dense = X @ W_hat.t()
        Y_fold = torch.cat([X, XP], dim=1) @ torch.cat([Uq, Vq], dim=1).t()
        torch.cuda.synchronize()
    finally:
        torch.backends.cuda.matmul.allow_tf32 = hp
    # oracle: the same codes and centres, fp64 throughout
    Xd = X.double().cpu().numpy()
    W_ref = ko.reconstruct(kd.unpack_codes(dec.codes_u, n).T, kd.unpack_codes(dec.codes_v, n).T,
                           dec.centres_u.double().cpu().numpy(), dec.centres_v.double().cpu().numpy(),
                           ko.sign_mask(spec.sign_seed, n))                # (n, m)
    Y_ref = Xd @ W_ref
    scale = np.abs(Y_ref).max()
    assert np.abs(Y_dense.double().cpu().numpy() - Y_ref).max() <= 1e-5 * scale
    assert np.abs(Y_fold.double().cpu().numpy() - Y_ref).max() <= 1e-5 * scale
    # and the quantised layer is close to the original one
    Y_orig = Xd @ w.double().cpu().numpy().T
    assert np.linalg.norm(Y_ref - Y_orig) <= 0.35 * np.linalg.norm(Y_orig)
