"""Randomized-Hadamard rotation (Sec. 4, Kashin-DCT+H) on the device against the
fp64 oracle, and the rotated pipeline: rotate, decompose (Algorithm 1) and code,
reconstruct, rotate back.

Tolerance: the fp32 butterfly network adds log2(b) <= 14 rounding levels on
values whose magnitude the orthonormal transform preserves, so the error is a few
units of 2^-24 of max|y|; the tests allow 2e-6 max|y| (entry-wise)."""

import numpy as np
import pytest

from oracle import kashin_oracle as ko
from paper_2609_11687_gb300 import synth
from tests import parity

pytestmark = pytest.mark.gpu

TOL = 2e-6


@pytest.fixture(scope="module")
def kd():
    import torch
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2609_11687_gb300 import build
    build.build()
    from paper_2609_11687_gb300 import kashin
    return kashin


def _status(torch):
    return torch.zeros(1, dtype=torch.int32, device="cuda")


def _check(y_dev, x_host, seed, inverse=False):
    ref = ko.randomized_hadamard(np.asarray(x_host, dtype=np.float64).T, seed, inverse=inverse).T
    y = y_dev.double().cpu().numpy()
    err = np.abs(y - ref).max() / np.abs(ref).max()
    assert err <= TOL, err


@pytest.mark.parametrize("n", [16, 32, 48, 64, 128, 256, 512, 768, 1024, 2048, 3072, 4096, 8192, 11008, 14336,
                               16384, 32768, 65536])
def test_rht_forward_inverse_all_block_sizes(kd, n):
    import torch
    m = 5 if n <= 16384 else 2
    g = torch.Generator().manual_seed(n)
    x = torch.randn((m, n), generator=g)
    seed = 1000 + n
    st = _status(torch)
    y = kd.rht(x.cuda(), seed, status=st)
    torch.cuda.synchronize()
    _check(y, x.numpy(), seed)
    z = kd.rht(y, seed, inverse=True, status=st)            # fp32 in: the staged path
    zh = kd.rht(y.half(), seed, inverse=True, status=st)    # fp16 in, staged
    yh = kd.rht(x.cuda().half(), seed, status=st)           # fp16 forward, staged
    torch.cuda.synchronize()
    assert st.item() == 0
    _check(zh, y.half().float().cpu().numpy(), seed, inverse=True)
    _check(yh, x.half().float().numpy(), seed)
    _check(z, y.cpu().numpy(), seed, inverse=True)
    np.testing.assert_allclose(z.cpu().numpy(), x.numpy(), rtol=0, atol=4 * TOL * float(x.abs().max()))


@pytest.mark.parametrize("dtype", ["f16", "bf16"])
def test_rht_half_inputs(kd, dtype):
    import torch
    td = torch.float16 if dtype == "f16" else torch.bfloat16
    x = (torch.randn((7, 4096), generator=torch.Generator().manual_seed(3)) * 0.02).to(td)
    y = kd.rht(x.cuda(), 9)
    torch.cuda.synchronize()
    _check(y, x.float().numpy(), 9)
    # strided rows (ld = 4096 + 64, still 16-byte aligned: staged, one copy per vector run)
    base = torch.zeros((7, 4160), dtype=td)
    base[:, :4096] = x
    y2 = kd.rht(base.cuda()[:, :4096], 9)
    torch.cuda.synchronize()
    assert torch.equal(y2, y)


def test_rht_strided_unaligned_inplace_and_empty(kd):
    import torch
    base = torch.randn((6, 800), generator=torch.Generator().manual_seed(4)).cuda()
    # ld = 800 > n = 768, and an odd start (not 16-byte aligned: scalar load path)
    x = base[:, 1:769]
    assert x.stride(0) == 800 and x.data_ptr() % 16 != 0
    y = kd.rht(x, 21)
    torch.cuda.synchronize()
    _check(y, x.cpu().numpy(), 21)
    # in place on an fp32 tensor: equal to the out-of-place result bit for bit
    w = base[:, :768].clone()
    ref = kd.rht(w, 21)
    kd.rht(w, 21, out=w)
    torch.cuda.synchronize()
    assert torch.equal(w, ref)
    # m = 0 enqueues nothing
    e = torch.empty((0, 256), device="cuda")
    assert kd.rht(e, 1).shape == (0, 256)


def test_rht_spike_flattens_outlier_channel(kd):
    """Incoherence: an outlier channel (one input index x20 in every vector, the
    synthetic outlier recipe) is spread over its block: max|y| / rms(y) drops."""
    import torch
    spec = synth.llama7b_layer(0)[0]
    import dataclasses
    w = synth.generate(dataclasses.replace(spec, M=64), device="cuda")
    y = kd.rht(w, 77)
    torch.cuda.synchronize()
    wf = w.float()
    before = (wf.abs().amax(1) / wf.pow(2).mean(1).sqrt()).mean().item()
    after = (y.abs().amax(1) / y.pow(2).mean(1).sqrt()).mean().item()
    assert after < 0.5 * before, (before, after)
    _check(y[:8], w[:8].float().cpu().numpy(), 77)


def test_rht_fullsize_sampled(kd):
    """Full Llama-2-7B gate matrix (11008 vectors of n = 4096, fp16) in one call;
    sampled rows against the oracle."""
    import torch
    spec = synth.llama7b_layer(0)[4]
    assert (spec.N, spec.M) == (4096, 11008)
    w = synth.generate(spec, device="cuda")
    y = kd.rht(w, 5)
    torch.cuda.synchronize()
    idx = synth.pair_aligned_sample(spec.M, 16, seed=1)
    _check(y[idx], w[idx].float().cpu().numpy(), 5)


@pytest.mark.parametrize("n,m", [(768, 9), (4096, 6), (11008, 4)])
def test_rotated_pipeline_parity_and_roundtrip(kd, n, m):
    """Kashin-DCT+H: rotate, decompose + code (parity against the oracle on the
    rotated input the device decomposed), reconstruct, rotate back; the rotated
    round trip reproduces the weights to the same error as the unrotated one."""
    import torch
    import dataclasses
    spec = dataclasses.replace(synth.llama7b_layer(3)[0], N=n, M=m)
    w = synth.generate(spec, device="cuda")
    rot_seed, sign_seed, iters = 4242, 17, 16
    wr = kd.rht(w, rot_seed)
    dev = parity.device_outputs(kd, wr, iters, sign_seed, trace=True)
    torch.cuda.synchronize()
    rep = parity.compare(wr.double().cpu().numpy().T, sign_seed, iters, dev)
    print(rep)
    rep.check()
    dec = kd.decompose(wr, iters, sign_seed)
    what_r = kd.reconstruct(dec, n, sign_seed)
    what = kd.rht(what_r, rot_seed, inverse=True)
    torch.cuda.synchronize()
    # orthogonal rotation: the quantisation error norm is the same in both bases
    e_rot = (what_r - wr).norm().item()
    e_back = (what - w.float()).norm().item()
    assert abs(e_rot - e_back) <= 1e-5 * e_rot
    # the point of the rotation: the outlier channel no longer dominates the codebook
    # (oracle at n = 768 / 4096: relative error 0.196 -> 0.129, 0.225 -> 0.122)
    plain = kd.reconstruct(kd.decompose(w, iters, sign_seed), n, sign_seed)
    torch.cuda.synchronize()
    e_plain = (plain - w.float()).norm().item()
    assert e_back < 0.8 * e_plain, (e_back, e_plain)
