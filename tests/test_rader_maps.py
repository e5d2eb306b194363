"""Host proof of the index maps behind the kernels' 43-point DFT (Rader's mapping split in
halves, `dft_prime_rader` in csrc/kd_math.cuh), with numpy standing in for the registers.

The kernel takes inputs in the order g^-q and outputs in the order g^m (g a primitive root
mod R), forms u_q = x(g^-q) + x(-g^-q) and (-1)^q (x(g^-q) - x(-g^-q)), and runs two
length-H cyclic convolutions (H = (R-1)/2 odd) through a prime-factor DFT of H = A B with
input index (B n1 + A n2) mod H and output index (B (B^-1 mod A) k1 + A (A^-1 mod B) k2)
mod H.  These tests rebuild exactly those maps and check the result against the DFT's
definition, so a wrong root, order, sign or CRT constant fails here without a GPU."""

import numpy as np
import pytest


def primitive_root(r):
    for g in range(2, r):
        if all(pow(g, e, r) != 1 for e in range(1, r - 1)):
            return g
    raise ValueError(r)


def smallest_factor(h):
    d = 2
    while d * d <= h:
        if h % d == 0:
            return d
        d += 1
    return h


def dft(x, sgn):
    n = len(x)
    k = np.arange(n)
    return np.exp(sgn * 2j * np.pi * np.outer(k, k) / n) @ x


def pfa(y, a, b, sgn):
    """The kernel's prime-factor DFT of length a*b (gcd 1, both prime)."""
    n = a * b
    ka = b * pow(b, a - 2, a) % n if a > 2 else b % n
    kb = a * pow(a, b - 2, b) % n if b > 2 else a % n
    t = np.zeros((a, b), complex)
    for n2 in range(b):
        t[:, n2] = dft(np.array([y[(b * n1 + a * n2) % n] for n1 in range(a)]), sgn)
    out = np.zeros(n, complex)
    for k1 in range(a):
        s = dft(t[k1], sgn)
        for k2 in range(b):
            out[(ka * k1 + kb * k2) % n] = s[k2]
    return out


def rader(x, r, direction):
    """The kernel's arithmetic order, in complex128: returns X_k = sum_n x_n w^(nk),
    w = exp(direction 2 pi i / r)."""
    h = (r - 1) // 2
    a = smallest_factor(h)
    b = h // a
    g = primitive_root(r)
    gi = pow(g, r - 2, r)
    q = np.arange(h)
    nq = np.array([pow(gi, int(i), r) for i in q])
    u = x[nq] + x[(r - nq) % r]
    w = np.where(q % 2 == 1, x[(r - nq) % r] - x[nq], x[nq] - x[(r - nq) % r])
    cj = np.cos(2 * np.pi * np.array([pow(g, j, r) for j in range(h)]) / r)
    sj = np.sin(2 * np.pi * np.array([pow(g, j, r) for j in range(h)]) / r)
    jj = np.where(np.arange(h) % 2 == 1, -sj, sj)
    chat, jhat = pfa(cj, a, b, -1) / h, pfa(jj, a, b, -1) / h
    uu, ww = pfa(u, a, b, -1), pfa(w, a, b, -1)
    out = np.zeros(r, complex)
    out[0] = x[0] + uu[0]
    uu = uu * chat
    uu[0] += x[0]
    ww = ww * jhat
    uu, ww = pfa(uu, a, b, +1), pfa(ww, a, b, +1)
    for m in range(h):
        k = pow(g, m, r)
        s = direction * (-1) ** m
        out[k] = uu[m] + s * 1j * ww[m]
        out[r - k] = uu[m] - s * 1j * ww[m]
    return out


def test_root_and_split_of_43():
    """g = 3 generates the units mod 43 (3^21 = -1), and H = 21 = 3 x 7 with the CRT
    output constants 7 and 15 the kernel's PFA uses."""
    assert primitive_root(43) == 3 and pow(3, 21, 43) == 42
    assert smallest_factor(21) == 3
    assert (7 * pow(7, 1, 3)) % 21 == 7 and (3 * pow(3, 5, 7)) % 21 == 15


@pytest.mark.parametrize("r", [43, 31])
@pytest.mark.parametrize("direction", [-1, +1])
def test_rader_equals_dft(r, direction):
    """R = 43 (H = 3 x 7, the compiled plan) and R = 31 (H = 3 x 5): the mapped
    computation equals the DFT's definition to rounding, both directions."""
    rng = np.random.default_rng(r)
    x = rng.standard_normal(r) + 1j * rng.standard_normal(r)
    assert np.abs(rader(x, r, direction) - dft(x, direction)).max() < 1e-11 * np.abs(x).sum()


def test_pfa_is_a_dft():
    """The prime-factor maps give the length-21 DFT itself (both signs)."""
    rng = np.random.default_rng(0)
    y = rng.standard_normal(21) + 1j * rng.standard_normal(21)
    for sgn in (-1, +1):
        assert np.abs(pfa(y, 3, 7, sgn) - dft(y, sgn)).max() < 1e-12 * np.abs(y).sum()


def test_zero_frequency_spectra_are_real():
    """C^_0 = -1/(2H) (the cosines of all nonzero residues sum to -1/2) and J^_0 is real:
    the kernel applies both as one real scale."""
    r, h = 43, 21
    g = primitive_root(r)
    cj = np.cos(2 * np.pi * np.array([pow(g, j, r) for j in range(h)]) / r)
    sj = np.sin(2 * np.pi * np.array([pow(g, j, r) for j in range(h)]) / r)
    jj = np.where(np.arange(h) % 2 == 1, -sj, sj)
    assert abs(cj.sum() / h + 0.5 / h) < 1e-14
    assert abs(pfa(jj, 3, 7, -1)[0].imag) < 1e-13


def test_a_wrong_sign_trick_is_caught():
    """Dropping the (-1)^q factor on the differences (a plausible slip) breaks equality."""
    r, h = 43, 21
    rng = np.random.default_rng(1)
    x = rng.standard_normal(r) + 1j * rng.standard_normal(r)
    g = primitive_root(r)
    gi = pow(g, r - 2, r)
    nq = np.array([pow(gi, i, r) for i in range(h)])
    w_bad = x[nq] - x[(r - nq) % r]                       # no alternating sign
    sj = np.sin(2 * np.pi * np.array([pow(g, j, r) for j in range(h)]) / r)
    jj = np.where(np.arange(h) % 2 == 1, -sj, sj)
    q_bad = pfa(pfa(w_bad, 3, 7, -1) * pfa(jj, 3, 7, -1) / h, 3, 7, +1)
    ref = dft(x, -1)
    # the true Q_m is (X(g^-m... )) recovered from the reference: Im-part combination
    k = np.array([pow(g, m, r) for m in range(h)])
    q_true = ((ref[k] - ref[(r - k) % r]) / (-2j)) * (-1) ** np.arange(h)
    assert np.abs(q_bad - q_true).max() > 1e-3 * np.abs(x).sum() / r
