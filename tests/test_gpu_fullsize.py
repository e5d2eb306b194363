"""Full-size parity: every matrix of the 7B-shaped workloads is decomposed whole,
in the launch configuration bench.py times (one kd_decompose per matrix, inputs
generated on the device); sampled vector pairs are then re-run with the trace on
a gathered copy (pairs kept whole, so the arithmetic is identical) and checked

  * bitwise against the full-size run (codes, centres, coefficients), and
  * against the CPU oracle with the tie-following protocol of tests/parity.py,
    including the per-vector residual norms ||r_k|| and the matrix's reconstruction
    error E = ||W - W_hat||_F / ||W||_F (kd_reconstruct on the device's codes).

The residual check runs at k = 4, 6, 8 as well as 16 on the bench's two vector
lengths, so every block index up to 16 is compared with the oracle where fp32
still resolves it; a device run stopped after 8 blocks must fail the k = 16 check.
"""

import dataclasses

import numpy as np
import pytest

from paper_2609_11687_gb300 import synth
from tests import parity

pytestmark = pytest.mark.gpu

ITERS = 16
SAMPLE_VECTORS = 256  # 128 pairs per matrix


def _cases():
    out = [("cfg3", s) for s in synth.config3()]
    out += [("cfg4", s) for s in synth.config4(layers=[31])]
    c5 = synth.config5(layers=[0, 31])
    out += [("cfg5", s) for s in c5 if s.name.startswith("pythia.L31") or s.name.startswith("mistral.L0")]
    return out


CASES = _cases()


@pytest.fixture(scope="module")
def kd():
    import torch
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2609_11687_gb300 import build
    build.build()
    from paper_2609_11687_gb300 import kashin
    return kashin


# the k-means refinement at full size too: the gate and down projections of the 7B layer
KM_CASES = [("cfg3-km3", s) for s in synth.config3() if s.name.endswith(("gate", "down"))]


def _run(kd, cfg, spec, kmeans_iters=0, iters=ITERS):
    import torch
    w = synth.generate(spec, device="cuda")                  # (M, N) fp16, device generator
    full = kd.decompose(w, iters, spec.sign_seed, coeffs=True, kmeans_iters=kmeans_iters)
    idx = synth.pair_aligned_sample(spec.M, SAMPLE_VECTORS, seed=spec.seed + 17)
    sub = w[idx].contiguous()
    dev = parity.device_outputs(kd, sub, iters, spec.sign_seed, trace=True, kmeans_iters=kmeans_iters,
                                w_hat=True)
    torch.cuda.synchronize()
    sel = torch.tensor(idx, device="cuda")
    for name in ("centres_u", "centres_v", "coeffs"):
        np.testing.assert_array_equal(getattr(full, name)[sel].cpu().numpy(), dev[name], err_msg=name)
    np.testing.assert_array_equal(full.codes_u[sel].cpu().numpy(), dev["words_u"])
    np.testing.assert_array_equal(full.codes_v[sel].cpu().numpy(), dev["words_v"])
    x = sub.double().cpu().numpy().T
    rep = parity.compare(x, spec.sign_seed, iters, dev, kmeans_iters=kmeans_iters)
    print(cfg, spec.name, iters, rep)
    rep.check()
    return sub, x, rep


@pytest.mark.parametrize("cfg,spec", CASES, ids=[f"{c}-{s.name}" for c, s in CASES])
def test_fullsize_sampled_parity(kd, cfg, spec):
    _run(kd, cfg, spec)


@pytest.mark.parametrize("cfg,spec", KM_CASES, ids=[f"{c}-{s.name}" for c, s in KM_CASES])
def test_fullsize_sampled_parity_kmeans(kd, cfg, spec):
    _run(kd, cfg, spec, kmeans_iters=3)


# the bench's two vector lengths (gate: n = 4096, down: n = 11008) at fewer blocks
BLOCK_CASES = [(k, s) for k in (4, 6, 8) for s in synth.config3() if s.name.endswith(("gate", "down"))]


@pytest.mark.parametrize("iters,spec", BLOCK_CASES, ids=[f"k{k}-{s.name}" for k, s in BLOCK_CASES])
def test_fullsize_sampled_parity_fewer_blocks(kd, iters, spec):
    _run(kd, "cfg3", spec, iters=iters)


@pytest.mark.parametrize("spec", [s for s in synth.config3() if s.name.endswith(("gate", "down"))],
                         ids=lambda s: s.name)
def test_truncated_run_fails_the_residual_check(kd, spec):
    """Self-check of the residual comparison: the device's k = 8 residuals set against
    the oracle's k = 16 ones (built on the host from two honest runs) must fail."""
    sub, x, rep16 = _run(kd, "cfg3", spec)
    d8 = kd.decompose(sub, 8, spec.sign_seed, factors=True)
    r8 = d8.resid.double().cpu().numpy().T
    nx = np.linalg.norm(x, axis=0)
    r8n = np.linalg.norm(r8, axis=0) / nx
    with pytest.raises(AssertionError):
        parity.check_residuals(r8n, rep16.r_ora)
    parity.check_residuals(rep16.r_gpu, rep16.r_ora)


def test_beyond_2_31_entries_int64_indexing(kd):
    """A matrix of more than 2^31 entries (n = 4096, m = 524,291 vectors, 4.3 GB of
    fp16): vectors at the far end, whose element offsets exceed 2^31, must come out
    bitwise equal to a decomposition of just those vectors.  Empty inputs are legal."""
    import torch
    n, m = 4096, (1 << 19) + 3
    assert n * m > 2**31
    g = torch.Generator(device="cuda").manual_seed(11)
    w = (torch.randn((m, n), generator=g, device="cuda", dtype=torch.float32) * 0.02).half()
    full = kd.decompose(w, 4, 5)
    idx = [0, 1, m - 5, m - 4, m - 3, m - 2, m - 1]
    sub = kd.decompose(w[idx[0]:idx[0] + 2].contiguous(), 4, 5)
    tail = kd.decompose(w[m - 5:].contiguous(), 4, 5)      # pairs (m-5, m-4), (m-3, m-2), (m-1)
    torch.cuda.synchronize()
    assert torch.equal(full.codes_u[:2], sub.codes_u) and torch.equal(full.centres_v[:2], sub.centres_v)
    assert torch.equal(full.codes_u[m - 5:], tail.codes_u) and torch.equal(full.codes_v[m - 5:], tail.codes_v)
    assert torch.equal(full.centres_u[m - 5:], tail.centres_u)
    del w, full
    # m = 0: nothing to do, no error
    e = torch.empty((0, n), dtype=torch.float16, device="cuda")
    out = kd.decompose(e, 4, 5)
    assert out.codes_u.shape == (0, n // 16)
    bat = kd.decompose_batch([e, e], 4, [1, 2])
    assert len(bat) == 2
