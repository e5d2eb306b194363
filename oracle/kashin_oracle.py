"""CPU oracle for the Kashin-DCT decomposition and 2-bit coding (TEST INFRASTRUCTURE).

This module is the slow, plain, obviously-correct reference that the CUDA path is
checked against.  It is test infrastructure: only ``tests/``,
``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline leg may import it, and
the library never calls it.  It shares no code with the CUDA path: no fast
transform, no factorisation, no tables.

Everything is float64 NumPy with an explicit ``N x N`` DCT-II matrix:

* ``dct2_matrix``          -- orthonormal DCT-II (Sec. 3.1, footnote on ``norm='ortho'``;
                              App. C footnote).  Row 0 carries the extra ``1/sqrt 2``
                              that makes the matrix orthogonal (the printed formula omits it).
* ``sign_mask``            -- the per-matrix sign set ``epsilon`` (Sec. 3.1 ``T_E``;
                              App. C: drawn once per layer from a fixed seed).  The paper
                              does not name its generator; the oracle takes it to be
                              SplitMix64 (Steele, Lea & Flood, OOPSLA 2014): bit 63 of
                              the mix of ``seed + (j + 1) * gamma`` set means -1.
* ``apply_p``              -- ``P z = IDCT(eps * DCT(z))`` with the dense matrix (Alg. 1).
* ``decompose``            -- Algorithm 1 (Greedy Algorithm with Alternating Updates)
                              written out step by step, with ``sign(0) = 0`` and the
                              step divisor ``N`` as printed.  Optional tie-follow.
* ``centres`` / ``codes``  -- the closed-form centres +-c1 +-c2 (Sec. 2.1) and the
                              nearest-centre 2-bit code (Sec. 2.1, App. C).
* ``kmeans_refine``        -- the few k-means refinement iterations that Sec. 2.1 runs
                              from the closed-form centres: 1-D Lloyd steps with 4
                              centres, an empty cluster keeps its centre.
* ``reconstruct``          -- dequantised ``W_hat = U_q + P V_q`` (App. C, Eq. 11).
* ``randomized_hadamard``  -- the randomized-Hadamard incoherence rotation that the
                              Kashin-DCT+H pipeline applies to a weight matrix before the
                              decomposition (Sec. 4): ``y = (I (x) H_b / sqrt b) diag(s) x``
                              per vector, Sylvester ``H_b`` on blocks of ``b`` = the largest
                              power of two dividing the length (at most 16384), signs ``s``
                              from the same SplitMix64 sequence as ``epsilon``.
* ``greedy_original``      -- Algorithm 2 (App. B), the original vector greedy algorithm
                              that Fig. 2 compares against: one projection step per
                              update on whichever of ``x`` and ``Q x`` has the larger
                              ``l_1`` norm.

Parity pins (tests/test_oracle_pins.py) tie each function to something the paper
or mathematics fixes; the ``l_inf`` bound constant of Theorem 2 contains the
unknown ``c_3`` and is *parity unpinned* as a number (only the coefficient-sum
form of the bound is checked).
"""

from __future__ import annotations

import dataclasses
from typing import Optional

import numpy as np

# ---------------------------------------------------------------------------
# Orthonormal DCT-II and the sign-randomised operator P (Sec. 3.1, App. C)
# ---------------------------------------------------------------------------


def dct2_matrix(N: int) -> np.ndarray:
    """Orthonormal DCT-II matrix ``C[j, n] = s_j sqrt(2/N) cos(pi (2n+1) j / (2N))``.

    ``s_0 = 1/sqrt(2)``, ``s_j = 1`` otherwise (Sec. 3.1 basis ``phi_j`` with the
    ``norm='ortho'`` convention of the footnote), so ``C^T = C^{-1}``.
    """
    n = np.arange(N, dtype=np.float64)[None, :]
    j = np.arange(N, dtype=np.float64)[:, None]
    C = np.sqrt(2.0 / N) * np.cos(np.pi * (2.0 * n + 1.0) * j / (2.0 * N))
    C[0, :] *= 1.0 / np.sqrt(2.0)
    return C


_MASK64 = (1 << 64) - 1
_GAMMA = 0x9E3779B97F4A7C15


def splitmix64(state: int) -> int:
    """SplitMix64 output function applied to a 64-bit state (Steele, Lea & Flood 2014)."""
    z = state & _MASK64
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & _MASK64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & _MASK64
    return z ^ (z >> 31)


def sign_mask(seed: int, N: int) -> np.ndarray:
    """``epsilon_j`` for DCT coefficient ``j`` (0-based): +1, or -1 where bit 63 of
    ``splitmix64(seed + (j + 1) * gamma)`` is set.  One mask per matrix, shared by
    all its columns (App. C)."""
    out = np.empty(N, dtype=np.float64)
    s = int(seed) & _MASK64
    for j in range(N):
        z = splitmix64((s + (j + 1) * _GAMMA) & _MASK64)
        out[j] = -1.0 if (z >> 63) else 1.0
    return out


def p_matrix(N: int, eps: np.ndarray) -> np.ndarray:
    """Dense ``P = C^T diag(eps) C`` (the operator U_{E,Phi} of Sec. 3.1)."""
    C = dct2_matrix(N)
    return C.T @ (eps[:, None] * C)


class POperator:
    """``P z = IDCT(eps * DCT(z))`` applied with the explicit DCT matrix (Alg. 1)."""

    def __init__(self, N: int, eps: np.ndarray):
        self.N = N
        self.eps = np.asarray(eps, dtype=np.float64)
        self.C = dct2_matrix(N)

    def __call__(self, z: np.ndarray) -> np.ndarray:
        z = np.asarray(z, dtype=np.float64)
        a = self.C @ z                       # DCT
        if a.ndim == 1:
            a = self.eps * a                 # T_eps
        else:
            a = self.eps[:, None] * a
        return self.C.T @ a                  # IDCT = DCT^T


# ---------------------------------------------------------------------------
# Algorithm 1: Greedy Algorithm with Alternating Updates
# ---------------------------------------------------------------------------


@dataclasses.dataclass
class Decomposition:
    u: np.ndarray          # (N, M)
    vhat: np.ndarray       # (N, M), P-domain factor; v = P vhat
    r: np.ndarray          # (N, M) residual r_k
    coeffs: np.ndarray     # (4, M): c1, c2 (block 0, steps 1-2), d1, d2 (block 0, steps 3-4)
    lambdas: np.ndarray    # (4k, M): coefficient of every atomic step
    step_norms: np.ndarray  # (4k + 1, M): ||rho||_2 entering each step, then final
    ties: int = 0          # decisions taken from the followed trace (|arg| <= tau)
    tie_flips: int = 0     # ... of which the followed sign differs from the oracle's own
    hard_mismatches: int = 0  # |arg| > tau but the followed sign differs (parity failure)


def _sign(a: np.ndarray) -> np.ndarray:
    """``sign`` with ``sign(0) = 0``: an exact zero entry takes no step (the paper does not say)."""
    return np.sign(a)


def decompose(x: np.ndarray, eps: np.ndarray, iters: int, follow: Optional[np.ndarray] = None,
              tau_abs: Optional[np.ndarray] = None, P: Optional[POperator] = None,
              follow_floor: Optional[np.ndarray] = None) -> Decomposition:
    """Run Algorithm 1 on every column of ``x`` (shape ``(N, M)``), float64.

    Per block t (k blocks): two greedy steps on the cube vertices Q_N update u,
    then two steps on P Q_N update vhat, exactly as Alg. 1 prints them::

        Delta_u    = sign(rho) * ||rho||_1 / N ;  u += Delta_u ;     rho -= Delta_u
        Delta_vhat = sign(P rho) * ||P rho||_1 / N ; vhat += Delta_vhat ; rho -= P Delta_vhat

    Tie-follow (test protocol for the discontinuous ``sign``): if ``follow`` is
    given (int8, shape ``(4k, N, M)``: the sign the device took at every atomic
    step, in natural element order), then wherever the oracle's own argument has
    ``|arg| <= tau_abs[col]`` the followed sign is used instead; a disagreement
    where ``|arg| > tau_abs`` is counted in ``hard_mismatches``.  Following only
    happens while the step's residual norm ``||rho||_2`` is at least
    ``follow_floor[col]`` (the device's rounding floor): below it the device's
    signs are rounding noise, so the oracle takes its own and counts nothing;
    each such step moves u or vhat by at most ``||rho||_2 / sqrt(N)``
    (Eq. lambda_bound).
    """
    x = np.asarray(x, dtype=np.float64)
    if x.ndim == 1:
        x = x[:, None]
    N, M = x.shape
    if P is None:
        P = POperator(N, eps)
    u = np.zeros_like(x)
    vhat = np.zeros_like(x)
    r = x.copy()
    coeffs = np.zeros((4, M))
    lambdas = np.zeros((4 * iters, M))
    norms = np.zeros((4 * iters + 1, M))
    stats = {"ties": 0, "flips": 0, "hard": 0}

    def choose_sign(arg: np.ndarray, step: int) -> np.ndarray:
        own = _sign(arg)
        if follow is None:
            return own
        dev = follow[step].astype(np.float64)
        near = np.abs(arg) <= tau_abs[None, :]
        if follow_floor is not None:
            resolved = np.linalg.norm(arg, axis=0) >= follow_floor
            dev = np.where(resolved[None, :], dev, own)
            near = near & resolved[None, :]
        stats["ties"] += int(near.sum())
        stats["flips"] += int((near & (dev != own)).sum())
        stats["hard"] += int((~near & (dev != own)).sum())
        return np.where(near, dev, own)

    step = 0
    for t in range(iters):
        rho = r.copy()
        for j in (1, 2):                     # two greedy steps from Q_N
            norms[step] = np.linalg.norm(rho, axis=0)
            lam = np.abs(rho).sum(axis=0) / N
            du = choose_sign(rho, step) * lam[None, :]
            u = u + du
            rho = rho - du
            lambdas[step] = lam
            if t == 0:
                coeffs[j - 1] = lam
            step += 1
        for j in (3, 4):                     # two greedy steps from P Q_N
            norms[step] = np.linalg.norm(rho, axis=0)
            y = P(rho)
            lam = np.abs(y).sum(axis=0) / N
            dv = choose_sign(y, step) * lam[None, :]
            vhat = vhat + dv
            rho = rho - P(dv)
            lambdas[step] = lam
            if t == 0:
                coeffs[j - 1] = lam
            step += 1
        r = rho
    norms[step] = np.linalg.norm(r, axis=0)
    return Decomposition(u=u, vhat=vhat, r=r, coeffs=coeffs, lambdas=lambdas, step_norms=norms,
                         ties=stats["ties"], tie_flips=stats["flips"], hard_mismatches=stats["hard"])


# ---------------------------------------------------------------------------
# Randomized-Hadamard incoherence rotation (Sec. 4, Kashin-DCT+H)
# ---------------------------------------------------------------------------

RHT_MAX_BLOCK = 16384


def hadamard_matrix(b: int) -> np.ndarray:
    """Sylvester Hadamard matrix of order ``b`` (a power of two):
    ``H_1 = [1]``, ``H_2k = [[H_k, H_k], [H_k, -H_k]]``."""
    assert b >= 1 and (b & (b - 1)) == 0
    H = np.ones((1, 1))
    while H.shape[0] < b:
        H = np.block([[H, H], [H, -H]])
    return H


def rht_block(n: int) -> int:
    """Block length of the rotation for vectors of length ``n``: the largest power
    of two dividing ``n``, capped at ``RHT_MAX_BLOCK``."""
    b = n & -n
    return min(b, RHT_MAX_BLOCK)


def randomized_hadamard(x: np.ndarray, seed: int, inverse: bool = False) -> np.ndarray:
    """Rotate every column of ``x`` (shape ``(n, m)`` or ``(n,)``), float64.

    Forward: ``y = R x`` with ``R = (I_{n/b} (x) H_b / sqrt(b)) diag(s)``: flip signs
    by ``s = sign_mask(seed, n)``, then an orthonormal Hadamard transform on each
    contiguous block of ``b = rht_block(n)`` entries.  Inverse: ``R^T``, i.e. the
    block transform first, then the sign flip (``H_b`` is symmetric).
    """
    x = np.asarray(x, dtype=np.float64)
    one = x.ndim == 1
    if one:
        x = x[:, None]
    n = x.shape[0]
    b = rht_block(n)
    Hn = hadamard_matrix(b) / np.sqrt(b)
    s = sign_mask(seed, n)[:, None]
    z = x if inverse else s * x
    y = np.empty_like(z)
    for k in range(n // b):
        y[k * b:(k + 1) * b] = Hn @ z[k * b:(k + 1) * b]
    if inverse:
        y = s * y
    return y[:, 0] if one else y


# ---------------------------------------------------------------------------
# Algorithm 2: the original vector greedy algorithm (App. B)
# ---------------------------------------------------------------------------


@dataclasses.dataclass
class GreedyOriginal:
    u: np.ndarray           # (N,)
    vhat: np.ndarray        # (N,), transform-domain factor; v = Q^T vhat
    r: np.ndarray           # (N,) residual
    norms: np.ndarray       # (updates + 1,): ||r||_2 before the first update, then after each
    branch: np.ndarray      # (updates,): 0 = u-update, 1 = vhat-update
    coeffs: np.ndarray      # (updates,): projection coefficient of every update


def greedy_original(x: np.ndarray, Q, tol: float = 0.0, max_updates: int = 64) -> GreedyOriginal:
    """Algorithm 2 on one vector ``x`` (float64) with the orthogonal operator ``Q``
    (a callable; Fig. 2 compares with the same sign-randomised DCT ``P``, so
    ``Q^T = Q``).  While ``||r|| >= tol`` and fewer than ``max_updates`` updates:

    * if ``||r||_1 > ||Q r||_1``: ``s = sign(r)``, ``pi = (r . s / ||s||^2) s``,
      ``u += pi``, ``r -= pi``;
    * else: ``s = sign(Q r)``, ``pi = ((Q r) . s / ||s||^2) s``, ``vhat += pi``,
      ``r -= Q^T pi``.

    The printed listing writes the second projection as ``pi_x(Sign(Q x))``, i.e. with
    ``x`` itself on the left of the inner product; it is taken here as the projection
    of ``Q x`` (the only choice that makes the step the least-squares move along
    ``Q^T s``, as the first branch is along ``s``).  ``||s||^2`` counts the non-zero
    entries, so an exact zero is left alone as in Alg. 1.
    """
    r = np.asarray(x, dtype=np.float64).copy()
    u = np.zeros_like(r)
    vhat = np.zeros_like(r)
    norms = [np.linalg.norm(r)]
    branch = []
    coeffs = []
    while norms[-1] >= tol and len(branch) < max_updates:
        y = Q(r)
        if np.abs(r).sum() > np.abs(y).sum():
            s = _sign(r)
            nnz = float(s @ s)
            c = float(r @ s) / nnz if nnz else 0.0
            u = u + c * s
            r = r - c * s
            branch.append(0)
        else:
            s = _sign(y)
            nnz = float(s @ s)
            c = float(y @ s) / nnz if nnz else 0.0
            vhat = vhat + c * s
            r = r - Q(c * s)
            branch.append(1)
        coeffs.append(c)
        norms.append(np.linalg.norm(r))
        if c == 0.0:
            break
    return GreedyOriginal(u=u, vhat=vhat, r=r, norms=np.array(norms), branch=np.array(branch, dtype=np.int8),
                          coeffs=np.array(coeffs))


# ---------------------------------------------------------------------------
# Closed-form centres and 2-bit codes (Sec. 2.1, App. C)
# ---------------------------------------------------------------------------


def centres(a1: np.ndarray, a2: np.ndarray) -> np.ndarray:
    """The four peaks +-a1 +-a2 of a factor after its two block-0 updates, ascending.

    Returns shape ``(M, 4)``: ``[-(a1+a2), -|a1-a2|, |a1-a2|, a1+a2]``."""
    a1 = np.asarray(a1, dtype=np.float64)
    a2 = np.asarray(a2, dtype=np.float64)
    outer = a1 + a2
    inner = np.abs(a1 - a2)
    return np.stack([-outer, -inner, inner, outer], axis=-1)


def codes(values: np.ndarray, cent: np.ndarray) -> np.ndarray:
    """Index of the nearest centre for every entry (ties to the lower index).

    ``values`` has shape ``(N, M)``, ``cent`` shape ``(M, 4)`` ascending.  The
    decision is taken in float32 (the precision the device decides in): both
    the values and the centre midpoints are rounded to float32 first.  Each
    boundary is the midpoint of two adjacent centres.
    """
    v32 = np.asarray(values, dtype=np.float32)
    c32 = np.asarray(cent, dtype=np.float64)
    b = np.stack([(c32[:, 0] + c32[:, 1]) / 2, (c32[:, 1] + c32[:, 2]) / 2,
                  (c32[:, 2] + c32[:, 3]) / 2], axis=-1).astype(np.float32)  # (M, 3)
    out = np.zeros(v32.shape, dtype=np.int64)
    for i in range(3):
        out += (v32 > b[None, :, i]).astype(np.int64)
    return out


def boundary_distance(values: np.ndarray, cent: np.ndarray) -> np.ndarray:
    """Distance of every entry to its nearest decision boundary (float64)."""
    c = np.asarray(cent, dtype=np.float64)
    b = np.stack([(c[:, 0] + c[:, 1]) / 2, (c[:, 1] + c[:, 2]) / 2, (c[:, 2] + c[:, 3]) / 2], axis=-1)
    v = np.asarray(values, dtype=np.float64)
    return np.min(np.abs(v[:, :, None] - b[None, :, :]), axis=-1)


def pack_codes(code: np.ndarray) -> np.ndarray:
    """Pack 2-bit codes of shape ``(N, M)`` into ``(M, ceil(N/16))`` uint32 words:
    entry i of a column sits at bits ``2 (i mod 16)`` of word ``i // 16``."""
    N, M = code.shape
    W = (N + 15) // 16
    out = np.zeros((M, W), dtype=np.uint64)
    for i in range(N):
        out[:, i // 16] |= (code[i, :].astype(np.uint64) & 3) << np.uint64(2 * (i % 16))
    return out.astype(np.uint32)


def unpack_codes(words: np.ndarray, N: int) -> np.ndarray:
    """Inverse of :func:`pack_codes`: returns ``(N, M)`` int64 codes."""
    words = np.asarray(words, dtype=np.uint64)
    M = words.shape[0]
    out = np.zeros((N, M), dtype=np.int64)
    for i in range(N):
        out[i, :] = (words[:, i // 16] >> np.uint64(2 * (i % 16))) & np.uint64(3)
    return out


def dequantise(code: np.ndarray, cent: np.ndarray) -> np.ndarray:
    """``c[code]`` per column: ``(N, M)`` codes with ``(M, 4)`` centres."""
    M = cent.shape[0]
    return np.asarray(cent, dtype=np.float64)[np.arange(M)[None, :], code]


def kmeans_refine(values: np.ndarray, cent: np.ndarray, iters: int, follow: Optional[np.ndarray] = None,
                  window: Optional[np.ndarray] = None):
    """Lloyd refinement of each column's 4 centres (Sec. 2.1: the closed-form centres
    initialise k-means, then a small number of refinement iterations run).

    Per iteration: every entry goes to its nearest centre (ties to the lower index,
    decided in float32 like :func:`codes`), then each centre becomes the float64
    mean of its entries; a centre with no entries keeps its value.  Returns the
    refined centres ``(M, 4)``, the final codes ``(N, M)`` and the number of followed
    and hard-mismatched assignments.

    ``follow`` (int, ``(iters, N, M)``) gives the device's assignment at each
    iteration; where an entry lies within ``window[col]`` of a boundary the
    device's code is used (both are nearest-centre within rounding)."""
    v = np.asarray(values, dtype=np.float64)
    c = np.array(cent, dtype=np.float64, copy=True)
    N, M = v.shape
    ties = hard = 0
    for it in range(iters):
        code = codes(v, c)
        if follow is not None:
            near = boundary_distance(v, c) <= window[None, :]
            dev = follow[it].astype(np.int64)
            ties += int((near & (dev != code)).sum())
            hard += int((~near & (dev != code)).sum())
            code = np.where(near, dev, code)
        for q in range(4):
            member = code == q
            cnt = member.sum(axis=0)
            tot = np.where(member, v, 0.0).sum(axis=0)
            c[:, q] = np.where(cnt > 0, tot / np.maximum(cnt, 1), c[:, q])
    return c, codes(v, c), ties, hard


def reconstruct(code_u: np.ndarray, code_v: np.ndarray, cent_u: np.ndarray, cent_v: np.ndarray,
                eps: np.ndarray) -> np.ndarray:
    """Dequantised weight ``W_hat = U_q + P V_q`` (App. C: dense re-materialisation)."""
    uq = dequantise(code_u, cent_u)
    vq = dequantise(code_v, cent_v)
    P = POperator(uq.shape[0], eps)
    return uq + P(vq)


@dataclasses.dataclass
class Quantised:
    dec: Decomposition
    centres_u: np.ndarray   # (M, 4)
    centres_v: np.ndarray   # (M, 4)
    codes_u: np.ndarray     # (N, M)
    codes_v: np.ndarray     # (N, M)


def quantise(x: np.ndarray, seed: int, iters: int, follow: Optional[np.ndarray] = None,
             tau_abs: Optional[np.ndarray] = None, kmeans_iters: int = 0) -> Quantised:
    """Decompose every column (Alg. 1), then code each factor with its closed-form
    centres (Sec. 2.1): u with (c1, c2), vhat with (d1, d2); ``kmeans_iters`` Lloyd
    refinement iterations from those centres (0 = the closed form alone)."""
    x = np.asarray(x, dtype=np.float64)
    eps = sign_mask(seed, x.shape[0])
    dec = decompose(x, eps, iters, follow=follow, tau_abs=tau_abs)
    cu = centres(dec.coeffs[0], dec.coeffs[1])
    cv = centres(dec.coeffs[2], dec.coeffs[3])
    if kmeans_iters > 0:
        cu, code_u, _, _ = kmeans_refine(dec.u, cu, kmeans_iters)
        cv, code_v, _, _ = kmeans_refine(dec.vhat, cv, kmeans_iters)
        return Quantised(dec=dec, centres_u=cu, centres_v=cv, codes_u=code_u, codes_v=code_v)
    return Quantised(dec=dec, centres_u=cu, centres_v=cv, codes_u=codes(dec.u, cu),
                     codes_v=codes(dec.vhat, cv))
