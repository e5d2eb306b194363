"""Checks the algebraic factorisation that the CUDA kernels implement, against
the oracle's dense ``P = C^T diag(eps) C`` (Sec. 3.1, App. C).

The kernels never form C.  They hold a vector in Makhoul's even/odd order
(J. Makhoul, "A fast cosine transform in one and two dimensions", IEEE TASSP
1980): ``v[n] = x[2n]``, ``v[N-1-n] = x[2n+1]``, pack two real vectors as one
complex vector ``z = v_a + i v_b``, and apply

    P' z = IDFT( M( DFT(z) ) ),
    M: Z'_k = e+_k Z_k + e-_k exp(i pi k / N) Z_{N-k},   e+-_k = (eps_k +- eps_{N-k}) / 2,
       Z'_0 = eps_0 Z_0,  Z'_{N/2} = eps_{N/2} Z_{N/2},

which equals the permuted ``P`` on each real part.  This file models that with
numpy's FFT (a library step) so the identity is pinned before any kernel runs.
"""

import numpy as np
import pytest

from oracle import kashin_oracle as ko


def makhoul_perm(N):
    """perm[p] = natural index held at Makhoul position p."""
    p = np.arange(N)
    return np.where(p < N // 2, 2 * p, 2 * (N - 1 - p) + 1)


def fast_p_packed(z, eps):
    N = z.shape[0]
    Z = np.fft.fft(z, axis=0)
    k = np.arange(N)
    km = (-k) % N
    ep = (eps + eps[km]) / 2
    em = (eps - eps[km]) / 2
    w = np.exp(1j * np.pi * k / N)
    Zp = ep[:, None] * Z + (em * w)[:, None] * Z[km]
    Zp[0] = eps[0] * Z[0]
    Zp[N // 2] = eps[N // 2] * Z[N // 2]
    return np.fft.ifft(Zp, axis=0)


@pytest.mark.parametrize("N", [2, 4, 6, 12, 256, 768, 1376])
def test_packed_fast_p_matches_dense(N):
    eps = ko.sign_mask(N + 3, N)
    rng = np.random.default_rng(N)
    a = rng.standard_normal((N, 3))
    b = rng.standard_normal((N, 3))
    perm = makhoul_perm(N)
    z = a[perm] + 1j * b[perm]
    out = fast_p_packed(z, eps)
    P = ko.p_matrix(N, eps)
    inv = np.empty(N, dtype=np.int64)
    inv[perm] = np.arange(N)
    np.testing.assert_allclose(out.real[inv], P @ a, atol=1e-12)
    np.testing.assert_allclose(out.imag[inv], P @ b, atol=1e-12)
