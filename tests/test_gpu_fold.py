"""kd_matmul_2bit: the layer product straight from the 2-bit planes (App. C,
Y = X U_q^T + (X P) V_q^T), against the fp64 oracle.

The oracle expands the device's codes and centres itself (oracle.dequantise) and
applies its own dense P to the rows of X, in fp64; the device runs kd_apply_p for XP
and the product kernel.  Both sides use the device's codes and centres: the product
is what is checked here (which codes a decomposition picks is the decomposition's
parity, checked elsewhere).  Tolerance: 1e-5 of max |Y| per batch row."""

import numpy as np
import pytest
import torch

from oracle import kashin_oracle as ko
from paper_2609_11687_gb300 import synth

pytestmark = pytest.mark.gpu

TOL = 1e-5


@pytest.fixture(scope="module")
def kd():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2609_11687_gb300 import build
    build.build()
    from paper_2609_11687_gb300 import kashin
    return kashin


_P = {}


def _oracle_y(kd, dec, n, seed, x64):
    """fp64: X U_q^T + (X P) V_q^T from the device's codes and centres."""
    cu = ko.dequantise(kd.unpack_codes(dec.codes_u, n).T, dec.centres_u.double().cpu().numpy())  # (n, m)
    cv = ko.dequantise(kd.unpack_codes(dec.codes_v, n).T, dec.centres_v.double().cpu().numpy())
    if (n, seed) not in _P:
        _P[(n, seed)] = ko.POperator(n, ko.sign_mask(seed, n))
    xp = _P[(n, seed)](x64.T).T                                              # rows of X times P
    return x64 @ cu + xp @ cv


def _run(kd, w, seed, batch, iters=16, gen_seed=0):
    m, n = w.shape
    dec = kd.decompose(w, iters, seed)
    g = torch.Generator(device="cuda").manual_seed(gen_seed)
    x = torch.randn((batch, n), generator=g, device="cuda", dtype=torch.float32)
    xp = kd.apply_p(x, seed)
    y = kd.matmul_2bit(dec, x, xp)
    torch.cuda.synchronize()
    y_ora = _oracle_y(kd, dec, n, seed, x.double().cpu().numpy())
    err = np.abs(y.double().cpu().numpy() - y_ora).max(axis=1)
    scale = np.abs(y_ora).max(axis=1)
    assert (err <= TOL * scale).all(), (err / scale).max()
    return dec, x, xp, y


@pytest.mark.parametrize("name", ["L0.q", "L0.gate", "L0.down"])
@pytest.mark.parametrize("batch", [1, 3, 4])
def test_matmul_2bit_7b_shapes(kd, name, batch):
    """The 7B layer's 4096 x 4096, 4096 x 11008 and 11008 x 4096 matrices, whole."""
    spec = {s.name: s for s in synth.config3()}[name]
    w = synth.generate(spec, device="cuda")
    _run(kd, w, spec.sign_seed, batch, gen_seed=batch)


@pytest.mark.parametrize("n,m,batch", [(768, 37, 6), (1000, 19, 5), (256, 1, 2), (16, 9, 1), (16384, 21, 3)])
def test_matmul_2bit_ragged(kd, n, m, batch):
    """Channel counts that leave a partial tile, a length with a partial last code word
    (run-time-length path), a single channel, the shortest and the longest lengths; batch
    chunks 2+2+2, 2+2+1, 2, 1 and 2+1."""
    g = torch.Generator(device="cuda").manual_seed(n + m)
    w = (torch.randn((m, n), generator=g, device="cuda") * 0.02).half()
    _run(kd, w, 7, batch)


def test_matmul_2bit_matches_reconstructed_weight(kd):
    """The folded product equals X W_hat^T with W_hat from kd_reconstruct (fp32, the
    load-time path), to fp32 rounding."""
    g = torch.Generator(device="cuda").manual_seed(2)
    w = (torch.randn((300, 4096), generator=g, device="cuda") * 0.02).half()
    dec, x, xp, y = _run(kd, w, 11, 2)
    wh = kd.reconstruct(dec, 4096, 11, dtype=torch.float32)
    ref = x.double() @ wh.double().T
    torch.cuda.synchronize()
    err = (y.double() - ref).abs().amax(dim=1)
    assert (err <= TOL * ref.abs().amax(dim=1)).all()


def test_matmul_2bit_deterministic_and_empty(kd):
    g = torch.Generator(device="cuda").manual_seed(3)
    w = (torch.randn((64, 512), generator=g, device="cuda") * 0.02).half()
    dec = kd.decompose(w, 8, 4)
    x = torch.randn((3, 512), generator=g, device="cuda")
    xp = kd.apply_p(x, 4)
    a = kd.matmul_2bit(dec, x, xp)
    b = kd.matmul_2bit(dec, x, xp)
    torch.cuda.synchronize()
    assert torch.equal(a, b)
    e = kd.matmul_2bit(dec, x[:0], xp[:0])
    assert e.shape == (0, 64)


def test_batched_calls_equal_single_calls(kd):
    """kd_apply_p_batch and kd_matmul_2bit_batch over a layer-like set of matrices (two
    vector lengths, ragged counts) reproduce the single calls bit for bit."""
    g = torch.Generator(device="cuda").manual_seed(9)
    shapes = [(37, 768, 3), (64, 768, 4), (5, 768, 5), (21, 11008, 6)]
    decs, xs, xps = [], [], []
    for m, n, seed in shapes:
        w = (torch.randn((m, n), generator=g, device="cuda") * 0.02).half()
        decs.append(kd.decompose(w, 4, seed))
        xs.append(torch.randn((3, n), generator=g, device="cuda"))
    xps = kd.apply_p_batch(xs[:3], [3, 4, 5]) + kd.apply_p_batch(xs[3:], [6])
    ys = kd.matmul_2bit_batch(decs, xs, xps)
    for (m, n, seed), d, x, xp, y in zip(shapes, decs, xs, xps, ys):
        xp1 = kd.apply_p(x, seed)
        y1 = kd.matmul_2bit(d, x, xp1)
        torch.cuda.synchronize()
        assert torch.equal(xp, xp1) and torch.equal(y, y1)


def test_matmul_2bit_strided_rows(kd):
    """Rows of x and xp with ldx > n (and misaligned by one element, so the inputs take
    the element-wise path) and of y with ldy > m give the same result as contiguous
    rows, bit for bit."""
    g = torch.Generator(device="cuda").manual_seed(12)
    m, n, b = 70, 1536, 3
    w = (torch.randn((m, n), generator=g, device="cuda") * 0.02).half()
    dec = kd.decompose(w, 6, 8)
    x = torch.randn((b, n), generator=g, device="cuda")
    xp = kd.apply_p(x, 8)
    ref = kd.matmul_2bit(dec, x, xp)
    for off in (0, 1):
        xs = torch.zeros((b, n + 40), device="cuda")
        ps = torch.zeros((b, n + 40), device="cuda")
        xs[:, off:off + n] = x
        ps[:, off:off + n] = xp
        ys = torch.full((b, m + 9), float("nan"), device="cuda")
        st = kd.kd_matmul_2bit(dec.codes_u.data_ptr(), dec.codes_v.data_ptr(), dec.centres_u.data_ptr(),
                               dec.centres_v.data_ptr(), n, m, xs[:, off:].data_ptr(), ps[:, off:].data_ptr(), b,
                               n + 40, ys.data_ptr(), m + 9, torch.cuda.current_stream().cuda_stream)
        assert st == kd.KD_OK
        torch.cuda.synchronize()
        assert torch.equal(ys[:, :m], ref)
        assert torch.isnan(ys[:, m:]).all()            # nothing written past m


@pytest.mark.parametrize("n,ms", [(768, (37, 0, 5)), (11008, (3, 6)), (1000, (2, 7))])
def test_prepared_p_equals_batched(kd, n, ms):
    """kd_prepare_p once, then kd_apply_p_prepared (twice, the tables reused) equals
    kd_apply_p_batch with the same seeds bit for bit: a batched plan with an empty
    matrix, the one-launch-per-matrix plan of n = 11008, the run-time-length path."""
    g = torch.Generator(device="cuda").manual_seed(n)
    xs = [torch.randn((m, n), generator=g, device="cuda") for m in ms]
    seeds = [11 * (i + 1) for i in range(len(ms))]
    ref = kd.apply_p_batch(xs, seeds)
    ws = kd.prepare_p(n, seeds)
    for _ in range(2):
        got = kd.apply_p_prepared(xs, ws)
        torch.cuda.synchronize()
        for a, b in zip(ref, got):
            assert torch.equal(a, b)

