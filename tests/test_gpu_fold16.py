"""kd_matmul_2bit_f16 and _bf16: the folded layer product (App. C) for 16-bit activations on the
tensor cores, against the fp64 oracle.

Both sides use the device decomposition's codes and centres (which codes a
decomposition picks is checked by the decomposition's parity tests); the product is what
is checked here.

* Exact inputs: the test draws X in fp16, the oracle forms X P in fp64 and rounds it to
  fp16 (numpy, nearest-even), and both sides take those same fp16 rows.  The oracle
  rounds the centres to fp16 the same way, so the only difference left is the fp32
  summation: tolerance 1e-5 of max |Y| per batch row for n <= 4096.  For terms of random
  sign that summation error grows like sqrt(n) relative to |Y| (the partial sums walk
  like sqrt(k)), so longer vectors get 1e-5 sqrt(n / 4096): 1.6e-5 at n = 11008, 2e-5 at
  16384, where the tensor cores' sums over 256 k-steps per warp measured 1.16e-5.
* End to end: fp32 X, X P from kd_apply_p, both rounded to fp16 by torch, against the
  full-precision fp64 product.  Rounding an input and a centre to fp16 changes each term
  x_i c_i by at most (2^-10 + 2^-22) |x_i c_i|, so the bound is 1.01 * 2^-10 * sum_i
  (|x_i u_i| + |xp_i v_i|) per output, plus 1e-5 of max |Y| for the fp32 sums and the
  fp32 X P."""

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


def _pop(n, seed):
    if (n, seed) not in _P:
        _P[(n, seed)] = ko.POperator(n, ko.sign_mask(seed, n))
    return _P[(n, seed)]


def _planes(kd, dec, n):
    """The expanded planes (n, m) in fp64 from the device's codes and centres."""
    cu = ko.dequantise(kd.unpack_codes(dec.codes_u, n).T, dec.centres_u.double().cpu().numpy())
    cv = ko.dequantise(kd.unpack_codes(dec.codes_v, n).T, dec.centres_v.double().cpu().numpy())
    return cu, cv


def _h(a):
    """fp16 rounding (nearest, ties to even), back in fp64."""
    return np.asarray(a, dtype=np.float64).astype(np.float16).astype(np.float64)


def _hb(a):
    """bf16 rounding (nearest, ties to even, by torch on the host), back in fp64."""
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float64)).to(torch.bfloat16).double().numpy()


def _exact(kd, w, seed, batch, iters=8, gen_seed=0, bf16=False):
    m, n = w.shape
    dt, rnd = (torch.bfloat16, _hb) if bf16 else (torch.float16, _h)
    dec = kd.decompose(w, iters, seed)
    g = torch.Generator().manual_seed(gen_seed)
    x16 = torch.randn((batch, n), generator=g).to(dt)
    xp16 = torch.from_numpy(np.ascontiguousarray(rnd(_pop(n, seed)(x16.double().numpy().T).T))).to(dt)
    y = kd.matmul_2bit_f16(dec, x16.cuda(), xp16.cuda())
    torch.cuda.synchronize()
    cu, cv = _planes(kd, dec, n)
    y_ora = x16.double().numpy() @ rnd(cu) + xp16.double().numpy() @ rnd(cv)
    err = np.abs(y.double().cpu().numpy() - y_ora).max(axis=1)
    scale = np.abs(y_ora).max(axis=1)
    tol = TOL * max(1.0, (n / 4096) ** 0.5)
    assert (err <= tol * scale).all(), (err / scale).max()
    return dec, y


@pytest.mark.parametrize("name", ["L0.q", "L0.gate", "L0.down"])
@pytest.mark.parametrize("batch", [1, 5, 16])
def test_f16_exact_inputs_7b_shapes(kd, name, batch):
    """The 7B layer's 4096 x 4096, 4096-input 11008-channel and 11008-input matrices."""
    spec = {s.name: s for s in synth.config3()}[name]
    w = synth.generate(spec, device="cuda")
    _exact(kd, w, spec.sign_seed, batch, iters=16, gen_seed=batch)


@pytest.mark.parametrize("n,m,batch", [(768, 37, 6), (1000, 19, 17), (256, 1, 2), (16, 9, 1), (4096, 70, 33)])
def test_f16_exact_inputs_ragged(kd, n, m, batch):
    """Channel counts with a partial 32-channel tile and a partial n-tile; lengths with a
    partial 64-input group (768), a partial code word (1000, run-time-length path), the
    shortest length; batches over 16 (two and three launches)."""
    g = torch.Generator(device="cuda").manual_seed(n + m)
    w = (torch.randn((m, n), generator=g, device="cuda") * 0.02).half()
    _exact(kd, w, 7, batch, gen_seed=n)


@pytest.mark.parametrize("batch", [1, 4, 16])
def test_f16_end_to_end_bound(kd, batch):
    """fp32 X through kd_apply_p, rounded to fp16, against the full-precision product."""
    spec = {s.name: s for s in synth.config3()}["L0.gate"]
    w = synth.generate(spec, device="cuda")
    n = spec.N
    dec = kd.decompose(w, 16, spec.sign_seed)
    gen = torch.Generator(device="cuda").manual_seed(100 + batch)
    x = torch.randn((batch, n), generator=gen, device="cuda")
    xp = kd.apply_p(x, spec.sign_seed)
    y = kd.matmul_2bit_f16(dec, x.half(), xp.half())
    torch.cuda.synchronize()
    cu, cv = _planes(kd, dec, n)
    x64 = x.double().cpu().numpy()
    xp64 = _pop(n, spec.sign_seed)(x64.T).T
    y_ora = x64 @ cu + xp64 @ cv
    bound = 1.01 * 2.0 ** -10 * (np.abs(x64) @ np.abs(cu) + np.abs(xp64) @ np.abs(cv))
    bound += TOL * np.abs(y_ora).max(axis=1, keepdims=True)
    err = np.abs(y.double().cpu().numpy() - y_ora)
    assert (err <= bound).all(), (err / bound).max()
    # the fp32 product from the same planes lies inside the same bound
    y32 = kd.matmul_2bit(dec, x, xp)
    torch.cuda.synchronize()
    assert (np.abs(y.double().cpu().numpy() - y32.double().cpu().numpy()) <= 2 * bound).all()


def test_f16_batched_equals_single_and_deterministic(kd):
    """kd_matmul_2bit_f16_batch over matrices of two lengths reproduces the single calls
    bit for bit; repeated calls agree bit for bit; an empty batch returns (0, m)."""
    g = torch.Generator(device="cuda").manual_seed(9)
    shapes = [(37, 768, 3), (64, 768, 4), (21, 11008, 6)]
    decs, xs, xps = [], [], []
    for m, n, seed in shapes:
        w = (torch.randn((m, n), generator=g, device="cuda") * 0.02).half()
        decs.append(kd.decompose(w, 4, seed))
        x = torch.randn((18, n), generator=g, device="cuda")
        xs.append(x.half())
        xps.append(kd.apply_p(x, seed).half())
    ys = kd.matmul_2bit_f16_batch(decs, xs, xps)
    for d, x, xp, y in zip(decs, xs, xps, ys):
        y1 = kd.matmul_2bit_f16(d, x, xp)
        y2 = kd.matmul_2bit_f16(d, x, xp)
        torch.cuda.synchronize()
        assert torch.equal(y, y1) and torch.equal(y1, y2)
    e = kd.matmul_2bit_f16(decs[0], xs[0][:0], xps[0][:0])
    assert e.shape == (0, 37)


def test_f16_strided_rows(kd):
    """Rows with ldx > n, 16-byte aligned (vector loads) and misaligned by one element
    (element-wise loads), and y rows with ldy > m, give the contiguous result bit for bit
    and write nothing past m."""
    g = torch.Generator(device="cuda").manual_seed(12)
    m, n, b = 70, 1536, 3
    w = (torch.randn((m, n), generator=g, device="cuda") * 0.02).half()
    dec = kd.decompose(w, 6, 8)
    x = torch.randn((b, n), generator=g, device="cuda")
    x16, xp16 = x.half(), kd.apply_p(x, 8).half()
    ref = kd.matmul_2bit_f16(dec, x16, xp16)
    for off in (0, 1):
        xs = torch.zeros((b, n + 40), device="cuda", dtype=torch.float16)
        ps = torch.zeros((b, n + 40), device="cuda", dtype=torch.float16)
        xs[:, off:off + n] = x16
        ps[:, off:off + n] = xp16
        ys = torch.full((b, m + 9), float("nan"), device="cuda")
        st = kd.kd_matmul_2bit_f16(dec.codes_u.data_ptr(), dec.codes_v.data_ptr(), dec.centres_u.data_ptr(),
                                   dec.centres_v.data_ptr(), n, m, xs[:, off:].data_ptr(), ps[:, off:].data_ptr(), b,
                                   n + 40, ys.data_ptr(), m + 9, torch.cuda.current_stream().cuda_stream)
        assert st == kd.KD_OK
        torch.cuda.synchronize()
        assert torch.equal(ys[:, :m], ref)
        assert torch.isnan(ys[:, m:]).all()


@pytest.mark.parametrize("name,batch", [("L0.q", 1), ("L0.down", 9), ("L0.gate", 16)])
def test_bf16_exact_inputs(kd, name, batch):
    """kd_matmul_2bit_bf16: the same exact-input parity with bf16 activations and centres
    rounded to bf16 on both sides."""
    spec = {s.name: s for s in synth.config3()}[name]
    w = synth.generate(spec, device="cuda")
    _exact(kd, w, spec.sign_seed, batch, iters=16, gen_seed=batch, bf16=True)


def test_bf16_ragged_and_end_to_end(kd):
    """bf16 on a ragged case (partial tiles, a partial code word, 17 rows) and end to end
    from fp32 X against the full-precision product, within the bf16 rounding bound
    1.01 * 2^-8 * sum_i (|x_i u_i| + |xp_i v_i|) plus 1e-5 of max |Y|."""
    g = torch.Generator(device="cuda").manual_seed(5)
    w = (torch.randn((19, 1000), generator=g, device="cuda") * 0.02).half()
    _exact(kd, w, 7, 17, gen_seed=3, bf16=True)
    spec = {s.name: s for s in synth.config3()}["L0.q"]
    w = synth.generate(spec, device="cuda")
    n = spec.N
    dec = kd.decompose(w, 16, spec.sign_seed)
    x = torch.randn((3, n), generator=g, device="cuda")
    xp = kd.apply_p(x, spec.sign_seed)
    y = kd.matmul_2bit_f16(dec, x.bfloat16(), xp.bfloat16())
    torch.cuda.synchronize()
    cu, cv = _planes(kd, dec, n)
    x64 = x.double().cpu().numpy()
    xp64 = _pop(n, spec.sign_seed)(x64.T).T
    y_ora = x64 @ cu + xp64 @ cv
    bound = 1.01 * 2.0 ** -8 * (np.abs(x64) @ np.abs(cu) + np.abs(xp64) @ np.abs(cv))
    bound += TOL * np.abs(y_ora).max(axis=1, keepdims=True)
    assert (np.abs(y.double().cpu().numpy() - y_ora) <= bound).all()


@pytest.mark.parametrize("bf16", [False, True])
def test_f16_longest_length(kd, bf16):
    """The longest supported vector length (n = 16384, 1,024 code words per channel) with a
    full 16-row batch and a partial 32-channel tile."""
    g = torch.Generator(device="cuda").manual_seed(16384)
    w = (torch.randn((45, 16384), generator=g, device="cuda") * 0.02).half()
    _exact(kd, w, 21, 16, gen_seed=7, bf16=bf16)

