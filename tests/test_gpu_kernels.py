"""GPU parity tests: the CUDA path through the C ABI against the CPU oracle."""

import numpy as np
import pytest

from oracle import kashin_oracle as ko
from paper_2609_11687_gb300 import synth
from tests import parity

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


@pytest.fixture(scope="module")
def torch_mod():
    import torch
    return torch


def _rand(torch, shape, seed, dtype=None, scale=0.02):
    g = torch.Generator().manual_seed(seed)
    x = torch.randn(shape, generator=g) * scale
    return x if dtype is None else x.to(dtype)


# ---------------------------------------------------------------------------
# The transform alone (K4): P via the fast path vs the dense oracle matrix
# ---------------------------------------------------------------------------

ALL_N = [16, 32, 64, 128, 256, 512, 768, 1024, 1536, 2048, 3072, 4096, 8192, 11008, 14336, 16384]


@pytest.mark.parametrize("n", ALL_N)
def test_apply_p_matches_dense(kd, torch_mod, n):
    torch = torch_mod
    m = 7  # odd: the last pair has one vector
    x = _rand(torch, (m, n), seed=n, scale=1.0)
    y = kd.apply_p(x.cuda(), sign_seed=n + 5).cpu().numpy().astype(np.float64)
    P = ko.POperator(n, ko.sign_mask(n + 5, n))
    ref = P(x.numpy().astype(np.float64).T).T
    rms = np.sqrt((x.numpy().astype(np.float64) ** 2).mean(axis=1, keepdims=True))
    err = np.abs(y - ref) / rms
    # fp32 FFT: error grows like eps_32 * log2(n); 1e-5 * rms leaves a wide margin
    assert err.max() < 1e-5, err.max()
    l2 = np.linalg.norm(y - ref, axis=1) / np.linalg.norm(ref, axis=1)
    assert l2.max() < 2e-6, l2.max()


@pytest.mark.parametrize("n", [256, 768, 4096, 11008])
def test_apply_p_is_involution(kd, torch_mod, n):
    torch = torch_mod
    x = _rand(torch, (4, n), seed=3, scale=1.0).cuda()
    y = kd.apply_p(kd.apply_p(x, 9), 9)
    assert (y - x).abs().max().item() < 2e-5


# ---------------------------------------------------------------------------
# Full decomposition parity
# ---------------------------------------------------------------------------

def _parity(kd, torch, G_cpu, seed, iters=ITERS, layout="rows", kmeans_iters=0):
    """G_cpu: (M, N) tensor (vector-major) on the CPU holding the exact inputs."""
    w = G_cpu.cuda()
    if layout == "columns":
        w = G_cpu.t().contiguous().cuda()
    dev = parity.device_outputs(kd, w, iters, seed, trace=True, layout=layout, kmeans_iters=kmeans_iters)
    x = G_cpu.to(torch.float64).numpy().T  # (N, M)
    rep = parity.compare(x, seed, iters, dev, kmeans_iters=kmeans_iters)
    return rep, dev


def test_config1_full(kd, torch_mod):
    torch = torch_mod
    spec = synth.config1()[0]
    G = synth.generate(spec)  # CPU generator, fp32 (256 vectors of 256)
    rep, _ = _parity(kd, torch, G, spec.sign_seed)
    print(rep)
    rep.check()


@pytest.mark.parametrize("iters", [0, 1, 2, 5])
def test_iteration_counts(kd, torch_mod, iters):
    torch = torch_mod
    G = _rand(torch, (9, 256), seed=iters + 10)
    rep, dev = _parity(kd, torch, G, 77, iters=iters)
    rep.check()
    if iters == 0:
        assert not dev["u"].any() and not dev["vhat"].any()
        np.testing.assert_array_equal(dev["resid"], G.numpy())
        assert not dev["words_u"].any() and not dev["words_v"].any()


@pytest.mark.parametrize("n,m", [(16, 3), (32, 7), (64, 5), (128, 5), (768, 13), (1024, 3), (1536, 5), (2048, 3),
                                 (3072, 9), (4096, 13), (8192, 3), (11008, 5), (14336, 3), (16384, 3)])
def test_shapes_ragged(kd, torch_mod, n, m):
    """Every compiled plan against the oracle, odd vector counts (a lone last vector)."""
    torch = torch_mod
    G = _rand(torch, (m, n), seed=n + m)
    rep, _ = _parity(kd, torch, G, seed=n)
    rep.check()


def test_single_vector(kd, torch_mod):
    torch = torch_mod
    G = _rand(torch, (1, 512), seed=1)
    rep, _ = _parity(kd, torch, G, seed=2)
    rep.check()


@pytest.mark.parametrize("kiters", [0, 3])
def test_zero_and_sparse_vectors(kd, torch_mod, kiters):
    """Degenerate vectors; with k-means on, the spike and constant vectors leave
    clusters empty (an empty cluster keeps its centre)."""
    torch = torch_mod
    G = _rand(torch, (6, 256), seed=4)
    G[1] = 0.0                           # all-zero vector
    G[2, ::3] = 0.0                      # exact zeros (fp16 underflow-like)
    G[3, :] = 0.0
    G[3, 17] = 0.5                       # a single spike
    G[4] = 1e-3                          # constant vector
    rep, dev = _parity(kd, torch, G, seed=5, kmeans_iters=kiters)
    rep.check(code_budget=False)   # the constant and spike vectors sit on boundaries by construction
    assert not dev["u"][1].any() and not dev["vhat"][1].any()
    assert not dev["centres_u"][1].any()
    assert not dev["words_u"][1].any()


def test_trace_and_factors_do_not_change_results(kd, torch_mod):
    torch = torch_mod
    w = _rand(torch, (10, 4096), seed=8, dtype=torch.float16).cuda()
    a = kd.decompose(w, ITERS, 3, factors=True, trace=True)
    b = kd.decompose(w, ITERS, 3, factors=False, coeffs=False, trace=False)
    torch.cuda.synchronize()
    for name in ("codes_u", "codes_v", "centres_u", "centres_v"):
        assert torch.equal(getattr(a, name), getattr(b, name)), name


def test_layouts_agree_bitwise(kd, torch_mod):
    torch = torch_mod
    G = _rand(torch, (11, 768), seed=12, dtype=torch.float16)
    a = kd.decompose(G.cuda(), ITERS, 4, factors=True)
    b = kd.decompose(G.t().contiguous().cuda(), ITERS, 4, layout="columns", factors=True)
    # leading dimension larger than the vector length
    padded = torch.zeros((11, 800), dtype=torch.float16)
    padded[:, :768] = G
    c = kd.decompose(padded.cuda()[:, :768], ITERS, 4, factors=True)
    torch.cuda.synchronize()
    for name in ("codes_u", "codes_v", "centres_u", "centres_v", "u", "vhat", "resid"):
        assert torch.equal(getattr(a, name), getattr(b, name)), name
        assert torch.equal(getattr(a, name), getattr(c, name)), name


def test_dtypes_agree_bitwise(kd, torch_mod):
    torch = torch_mod
    G16 = _rand(torch, (5, 4096), seed=21, dtype=torch.float16)
    Gb = _rand(torch, (5, 4096), seed=22, dtype=torch.bfloat16)
    for G in (G16, Gb):
        a = kd.decompose(G.cuda(), ITERS, 6, factors=True)
        b = kd.decompose(G.float().cuda(), ITERS, 6, factors=True)
        torch.cuda.synchronize()
        for name in ("codes_u", "codes_v", "centres_u", "u", "vhat"):
            assert torch.equal(getattr(a, name), getattr(b, name)), name


def test_nonfinite_input_sets_status(kd, torch_mod):
    torch = torch_mod
    w = _rand(torch, (4, 256), seed=1).cuda()
    ws = kd.Workspace(256)
    kd.decompose(w, 4, 0, workspace=ws)
    assert kd.read_status(ws) == kd.KD_OK
    w[2, 7] = float("nan")
    kd.decompose(w, 4, 0, workspace=ws)
    assert kd.read_status(ws) == kd.KD_ERR_NONFINITE
    w[2, 7] = float("inf")
    kd.decompose(w, 4, 0, workspace=ws)
    assert kd.read_status(ws) == kd.KD_ERR_NONFINITE
    w[2, 7] = 0.0
    kd.decompose(w, 4, 0, workspace=ws)
    assert kd.read_status(ws) == kd.KD_OK


def test_read_status_decodes_the_word(kd, torch_mod):
    """kd_read_status decodes the workspace's status word: bit 1 (a staged-input wait
    that expired) reads as KD_ERR_TIMEOUT, also together with bit 0; bit 0 alone as
    KD_ERR_NONFINITE; and the next decomposition clears the word.  The bits are written
    into the word directly: no wait is made to expire."""
    torch = torch_mod
    ws = kd.Workspace(256)
    word = ws.buf[:4].view(torch.int32)
    for bits, want in ((2, kd.KD_ERR_TIMEOUT), (3, kd.KD_ERR_TIMEOUT), (1, kd.KD_ERR_NONFINITE), (0, kd.KD_OK)):
        word.fill_(bits)
        assert kd.read_status(ws) == want
    word.fill_(2)
    kd.decompose(_rand(torch, (4, 256), seed=2).cuda(), 4, 0, workspace=ws)
    assert kd.read_status(ws) == kd.KD_OK


def test_deterministic(kd, torch_mod):
    torch = torch_mod
    w = _rand(torch, (64, 4096), seed=31, dtype=torch.float16).cuda()
    a = kd.decompose(w, ITERS, 1)
    b = kd.decompose(w, ITERS, 1)
    torch.cuda.synchronize()
    assert torch.equal(a.codes_u, b.codes_u) and torch.equal(a.centres_v, b.centres_v)


# ---------------------------------------------------------------------------
# k-means refinement of the centres (Sec. 2.1)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("n,m,kiters", [(256, 16, 3), (768, 9, 1), (3072, 6, 3), (4096, 10, 5), (11008, 4, 3)])
def test_kmeans_refinement_parity(kd, torch_mod, n, m, kiters):
    torch = torch_mod
    G = _rand(torch, (m, n), seed=n + 3, dtype=torch.float16)
    rep, dev = _parity(kd, torch, G.float(), seed=n, kmeans_iters=kiters)
    print(rep)
    rep.check()
    # refinement lowers each factor's within-cluster squared error vs the closed form
    closed = kd.decompose(G.cuda(), ITERS, n, factors=True)
    torch.cuda.synchronize()
    def sse(vals, cent, words):
        code = kd.unpack_codes(words, n)
        c = cent.cpu().numpy().astype(np.float64)
        return ((vals.cpu().numpy().astype(np.float64) - c[np.arange(m)[:, None], code]) ** 2).sum(1)
    assert np.all(sse(closed.u, torch.from_numpy(dev["centres_u"]), torch.from_numpy(dev["words_u"]))
                  <= sse(closed.u, closed.centres_u, closed.codes_u) * (1 + 1e-5))


def test_kmeans_zero_iters_is_closed_form(kd, torch_mod):
    torch = torch_mod
    w = _rand(torch, (6, 4096), seed=2, dtype=torch.float16).cuda()
    a = kd.decompose(w, ITERS, 5)
    b = kd.decompose(w, ITERS, 5, kmeans_iters=0)
    c = kd.decompose(w, ITERS, 5, kmeans_iters=2)
    torch.cuda.synchronize()
    assert torch.equal(a.centres_u, b.centres_u) and torch.equal(a.codes_v, b.codes_v)
    assert not torch.equal(a.centres_u, c.centres_u)


# ---------------------------------------------------------------------------
# Reconstruction (App. C dense re-materialisation)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("n", [256, 768, 4096])
def test_reconstruct_matches_oracle(kd, torch_mod, n):
    torch = torch_mod
    G = _rand(torch, (6, n), seed=n, dtype=torch.float16)
    dec = kd.decompose(G.cuda(), ITERS, 7)
    W = kd.reconstruct(dec, n, 7).cpu().numpy().astype(np.float64)      # (m, n)
    code_u = kd.unpack_codes(dec.codes_u, n).T
    code_v = kd.unpack_codes(dec.codes_v, n).T
    ref = ko.reconstruct(code_u, code_v, dec.centres_u.cpu().numpy(), dec.centres_v.cpu().numpy(),
                         ko.sign_mask(7, n)).T
    scale = np.abs(ref).max(axis=1, keepdims=True)
    assert (np.abs(W - ref) / scale).max() < 5e-6
    # quantisation error is a few per cent of the weight norm for 2+2 bits
    Gd = G.double().numpy()
    E = np.linalg.norm(Gd - W, axis=1) / np.linalg.norm(Gd, axis=1)
    assert E.max() < 0.5
    # output dtypes / layouts
    Wh = kd.reconstruct(dec, n, 7, dtype=torch.float16)
    Wc = kd.reconstruct(dec, n, 7, layout="columns")
    assert torch.allclose(Wh.float().cpu(), torch.from_numpy(W).float(), atol=1e-3, rtol=1e-3)
    assert torch.equal(Wc.t().cpu(), torch.from_numpy(W).float())


# ---------------------------------------------------------------------------
# Config 2: OPT-125M-shaped layer 0, every vector
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("mi", range(6))
def test_config2_layer0_all_vectors(kd, torch_mod, mi):
    torch = torch_mod
    spec = synth.config2(layers=[0])[mi]
    G = synth.generate(spec)  # CPU generator, fp16 (M, N)
    rep, _ = _parity(kd, torch, G, spec.sign_seed)
    print(spec.name, rep)
    rep.check()


def test_calls_only_enqueue_on_the_given_stream(kd, torch_mod):
    """The C ABI validates, enqueues on the caller's stream and returns: right after
    the call the stream's work (a ~4 ms decomposition) is still pending, and the
    results are there once that stream is synchronised."""
    torch = torch_mod
    from paper_2609_11687_gb300 import synth
    spec = synth.llama7b_layer(0)[4]                      # 11008 vectors of n = 4096
    w = synth.generate(spec, device="cuda")
    ws = kd.Workspace(spec.N)
    ref = kd.decompose(w, ITERS, spec.sign_seed, workspace=ws)
    torch.cuda.synchronize()
    s = torch.cuda.Stream()
    out = kd.Decomposed(codes_u=torch.zeros_like(ref.codes_u), codes_v=torch.zeros_like(ref.codes_v),
                        centres_u=torch.zeros_like(ref.centres_u), centres_v=torch.zeros_like(ref.centres_v),
                        coeffs=None, u=None, vhat=None, resid=None, trace=None)
    ws2 = kd.Workspace(spec.N)
    torch.cuda.synchronize()
    kd.decompose(w, ITERS, spec.sign_seed, workspace=ws2, out=out, stream=s)
    done = torch.cuda.Event()
    done.record(s)
    assert not done.query()          # still running: the call did not wait for it
    s.synchronize()
    assert done.query()
    assert torch.equal(out.codes_u, ref.codes_u) and torch.equal(out.centres_v, ref.centres_v)
