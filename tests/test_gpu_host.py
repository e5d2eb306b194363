"""kd_decompose_batch_host: host matrices in, host codes and centres out, through the C
ABI on one stream.  The outputs must equal the device-buffer batched call bit for bit
(the same kernel runs on staged copies of the same bytes)."""

import pytest
import torch

from paper_2609_11687_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def kd():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2609_11687_gb300 import build
    build.build()
    from paper_2609_11687_gb300 import kashin
    return kashin


def _check(kd, mats, seeds, iters=16, layout="rows", kmeans_iters=0):
    n = mats[0].shape[1] if layout == "rows" else mats[0].shape[0]
    host = [w.cpu().pin_memory() for w in mats]
    outs = [kd.host_outputs(w.shape[0] if layout == "rows" else w.shape[1], n, coeffs=True) for w in host]
    staging = torch.empty(kd.staging_size_host(host, layout, coeffs=True), dtype=torch.uint8, device="cuda")
    ws = kd.Workspace(n, count=len(host))
    stream = torch.cuda.current_stream()
    kd.decompose_batch_host(host, iters, seeds, outs, staging, ws, layout=layout, stream=stream,
                            kmeans_iters=kmeans_iters)
    ref = kd.decompose_batch([w.cuda() for w in mats], iters, seeds, layout=layout, coeffs=True,
                             kmeans_iters=kmeans_iters)
    torch.cuda.synchronize()
    for o, r in zip(outs, ref):
        for name in ("codes_u", "codes_v", "centres_u", "centres_v", "coeffs"):
            assert torch.equal(getattr(o, name), getattr(r, name).cpu()), name


def test_host_batch_equals_device_batch_7b_shapes(kd):
    """The 7B layer's q projection and down projection (n = 4096 in one launch, n = 11008
    one launch per matrix), fp16 rows, sampled to keep the test short."""
    specs = {s.name: s for s in synth.config3()}
    for names in (("L0.q", "L0.k"), ("L0.down",)):
        mats, seeds = [], []
        for nm in names:
            w = synth.generate(specs[nm], device="cuda")[:301].contiguous()
            mats.append(w)
            seeds.append(specs[nm].sign_seed)
        _check(kd, mats, seeds)


def test_host_batch_columns_and_refinement(kd):
    g = torch.Generator().manual_seed(3)
    mats = [(torch.randn((768, 37), generator=g) * 0.02).to(torch.bfloat16),
            (torch.randn((768, 64), generator=g) * 0.02).to(torch.bfloat16)]
    _check(kd, mats, [5, 6], iters=8, layout="columns", kmeans_iters=2)


def test_host_batch_empty_matrix(kd):
    g = torch.Generator().manual_seed(4)
    mats = [(torch.randn((6, 256), generator=g) * 0.02).half(), torch.empty((0, 256), dtype=torch.float16)]
    _check(kd, mats, [1, 2], iters=4)
