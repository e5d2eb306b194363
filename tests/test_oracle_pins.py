"""Pins for the CPU oracle: each function is tied to something the paper or the
mathematics fixes, independently of the oracle's own formulas.

* orthonormal DCT-II (Sec. 3.1 footnote): brute-force orthogonality, constant and
  single-cosine closed forms, SciPy's ``dct(norm='ortho')`` special case;
* P = IDCT o T_eps o DCT (Sec. 3.1, App. C): symmetric involution, N = 2 closed forms;
* sign mask: published SplitMix64 reference sequence;
* Algorithm 1: per-step identity Eq. (one_step), exact reconstruction, monotone
  residual (non-expansive steps, App. D), coefficient bounds Eq. (lambda_bound) and
  Eq. (uk_inf_naive), four values after one block (Sec. 2.1), hand-worked N = 4 and
  N = 2 cases with closed forms over k blocks;
* centres / codes / packing: hand-worked centres and exhaustive boundary cases.
"""

import numpy as np
import pytest

from oracle import kashin_oracle as ko
from tests.conftest import read_golden

# ---------------------------------------------------------------------------
# DCT-II
# ---------------------------------------------------------------------------


@pytest.mark.parametrize("N", [2, 3, 4, 8, 12, 43, 256])
def test_dct_orthogonal_bruteforce(N):
    C = ko.dct2_matrix(N)
    # brute force: every pair of rows, explicit dot products
    for a in range(min(N, 48)):
        for b in range(min(N, 48)):
            dot = sum(C[a, n] * C[b, n] for n in range(N))
            assert abs(dot - (1.0 if a == b else 0.0)) < 1e-12


@pytest.mark.parametrize("N", [4, 12, 256, 768])
def test_dct_of_constant_is_sqrtN_e0(N):
    X = ko.dct2_matrix(N) @ np.ones(N)
    expect = np.zeros(N)
    expect[0] = np.sqrt(N)
    np.testing.assert_allclose(X, expect, atol=1e-11)


@pytest.mark.parametrize("N,k0", [(8, 3), (43, 7), (256, 100)])
def test_dct_single_cosine(N, k0):
    # x_n = cos(pi (2n+1) k0 / 2N) is basis vector k0 scaled by sqrt(N/2)
    n = np.arange(N)
    x = np.cos(np.pi * (2 * n + 1) * k0 / (2 * N))
    X = ko.dct2_matrix(N) @ x
    expect = np.zeros(N)
    expect[k0] = np.sqrt(N / 2.0)
    np.testing.assert_allclose(X, expect, atol=1e-11)


@pytest.mark.parametrize("N", [16, 43, 768, 3072])
def test_dct_matches_scipy_ortho(N):
    fft = pytest.importorskip("scipy.fft")
    x = np.random.default_rng(N).standard_normal((N, 3))
    np.testing.assert_allclose(ko.dct2_matrix(N) @ x, fft.dct(x, type=2, norm="ortho", axis=0),
                               rtol=0, atol=1e-11)


# ---------------------------------------------------------------------------
# P
# ---------------------------------------------------------------------------


@pytest.mark.parametrize("N", [2, 3, 8, 43, 256])
def test_p_symmetric_involution(N):
    P = ko.p_matrix(N, ko.sign_mask(7, N))
    I = np.eye(N)
    assert np.abs(P - P.T).max() < 1e-13
    assert np.abs(P @ P - I).max() < 1e-13
    assert np.abs(P @ P.T - I).max() < 1e-13


def test_p_n2_closed_forms():
    swap = np.array([[0.0, 1.0], [1.0, 0.0]])
    assert np.abs(ko.p_matrix(2, np.array([1.0, -1.0])) - swap).max() < 1e-15
    assert np.abs(ko.p_matrix(2, np.array([1.0, 1.0])) - np.eye(2)).max() < 1e-15
    assert np.abs(ko.p_matrix(2, np.array([-1.0, -1.0])) + np.eye(2)).max() < 1e-15


def test_p_operator_matches_matrix():
    N = 43
    eps = ko.sign_mask(3, N)
    z = np.random.default_rng(0).standard_normal((N, 4))
    np.testing.assert_allclose(ko.POperator(N, eps)(z), ko.p_matrix(N, eps) @ z, atol=1e-13)


def test_all_plus_signs_give_identity():
    N = 12
    np.testing.assert_allclose(ko.p_matrix(N, np.ones(N)), np.eye(N), atol=1e-14)


# ---------------------------------------------------------------------------
# Sign mask
# ---------------------------------------------------------------------------


def test_splitmix64_reference_sequence():
    _, bare = read_golden("splitmix64_state0.txt")
    expect = [int(h, 16) for h in bare]
    state = 0
    for e in expect:
        state = (state + 0x9E3779B97F4A7C15) & ((1 << 64) - 1)
        assert ko.splitmix64(state) == e
    # epsilon_j is bit 63 of output j of the sequence started at the seed
    eps = ko.sign_mask(0, len(expect))
    assert list(eps) == [-1.0 if e >> 63 else 1.0 for e in expect]


def test_sign_mask_seed_dependence():
    a = ko.sign_mask(1, 512)
    b = ko.sign_mask(2, 512)
    assert set(np.unique(a)) == {-1.0, 1.0}
    assert (a != b).mean() > 0.3


# ---------------------------------------------------------------------------
# Algorithm 1
# ---------------------------------------------------------------------------


def _gauss(N, M, seed=0):
    return np.random.default_rng(seed).standard_normal((N, M)) * 0.02


@pytest.mark.parametrize("N", [8, 43, 256])
def test_step_identity_eq_one_step(N):
    """Eq. (one_step): ||y - lambda* w*||^2 = ||y||^2 - ||y||_1^2 / N, for every
    atomic step (u-steps directly, vhat-steps through the orthogonal P)."""
    x = _gauss(N, 5, seed=N)
    eps = ko.sign_mask(11, N)
    d = ko.decompose(x, eps, 4)
    n2 = d.step_norms ** 2
    drop = N * d.lambdas ** 2            # ||rho||_1^2 / N with lambda = ||rho||_1 / N
    np.testing.assert_allclose(n2[1:], n2[:-1] - drop, rtol=1e-9, atol=1e-14 * n2[0].max())


@pytest.mark.parametrize("N", [8, 43, 256])
def test_exact_reconstruction(N):
    x = _gauss(N, 6, seed=N + 1)
    eps = ko.sign_mask(5, N)
    d = ko.decompose(x, eps, 6)
    P = ko.p_matrix(N, eps)
    err = np.linalg.norm(x - d.u - P @ d.vhat - d.r, axis=0) / np.linalg.norm(x, axis=0)
    assert err.max() < 1e-12


def test_residual_monotone_and_decays():
    N = 256
    x = _gauss(N, 8, seed=3)
    d = ko.decompose(x, ko.sign_mask(0, N), 8)
    assert np.all(np.diff(d.step_norms, axis=0) <= 1e-15)
    blocks = d.step_norms[::4]
    ratio = blocks[1:] / blocks[:-1]
    assert np.all(ratio < 1.0)
    assert blocks[-1].max() / blocks[0].min() < 1e-4   # geometric decay (Theorem 2, first line)


@pytest.mark.parametrize("N", [43, 256])
def test_coefficient_bounds(N):
    """Eq. (lambda_bound): |lambda| <= ||rho||_2 / sqrt(N); Eq. (uk_inf_naive):
    ||u_k||_inf <= sum of the u-step |lambda|, same for vhat."""
    x = _gauss(N, 5, seed=N + 2)
    d = ko.decompose(x, ko.sign_mask(9, N), 5)
    assert np.all(d.lambdas <= d.step_norms[:-1] / np.sqrt(N) * (1 + 1e-12))
    lam = d.lambdas.reshape(-1, 4, d.lambdas.shape[1])
    assert np.all(np.abs(d.u).max(0) <= lam[:, 0:2].sum((0, 1)) * (1 + 1e-12))
    assert np.all(np.abs(d.vhat).max(0) <= lam[:, 2:4].sum((0, 1)) * (1 + 1e-12))


def test_four_peaks_after_one_block():
    """Sec. 2.1: after the two u-updates u takes only the values +-c1 +-c2; the
    same holds for vhat with d1, d2."""
    N = 256
    x = _gauss(N, 4, seed=5)
    d = ko.decompose(x, ko.sign_mask(1, N), 1)
    for col in range(4):
        c1, c2, d1, d2 = d.coeffs[:, col]
        allowed_u = np.array([c1 + c2, c1 - c2, -c1 + c2, -c1 - c2])
        allowed_v = np.array([d1 + d2, d1 - d2, -d1 + d2, -d1 - d2])
        assert np.min(np.abs(d.u[:, col][:, None] - allowed_u[None]), axis=1).max() < 1e-15
        assert np.min(np.abs(d.vhat[:, col][:, None] - allowed_v[None]), axis=1).max() < 1e-15


def test_hand_worked_n4_u_steps_and_centres():
    g, _ = read_golden("hand_n4_block0_u.txt")
    x = np.array(g["x"])
    d = ko.decompose(x, ko.sign_mask(0, 4), 1)
    assert d.coeffs[0, 0] == g["c1"][0] and d.coeffs[1, 0] == g["c2"][0]
    np.testing.assert_allclose(d.step_norms[:3, 0] ** 2, g["norm2"], rtol=1e-15)
    # u after one block = u after its two u-steps (the vhat-steps do not touch u)
    np.testing.assert_array_equal(d.u[:, 0], g["u2"])
    cent = ko.centres(np.array([g["c1"][0]]), np.array([g["c2"][0]]))
    np.testing.assert_array_equal(cent[0], g["centres"])
    b = g["boundaries"]
    vals = np.array([b[0], b[1], b[2], -10, -1, 1, 10], dtype=np.float64)[:, None]
    np.testing.assert_array_equal(ko.codes(vals, cent)[:, 0], [0, 1, 2, 0, 1, 2, 3])


def test_hand_worked_n2_swap_closed_form():
    g, _ = read_golden("hand_n2_swap.txt")
    x = np.array(g["x"])[:, None]
    swap = lambda z: np.asarray(z)[::-1].copy()   # exact P for eps = (+1, -1), N = 2
    for k in (1, 2, 5):
        d = ko.decompose(x, np.array(g["eps"]), k, P=swap)
        S = sum(16.0 ** -t for t in range(k))
        np.testing.assert_allclose(d.lambdas[:4, 0], g["lambda"], rtol=0, atol=0)
        np.testing.assert_allclose(d.u[:, 0], [0.75 * S, 0.0], rtol=1e-15, atol=0)
        np.testing.assert_allclose(d.vhat[:, 0], [0.0, 0.1875 * S], rtol=1e-15, atol=0)
        np.testing.assert_allclose(d.r[:, 0], [16.0 ** -k, 0.0], rtol=1e-15, atol=0)
        if k == 1:
            assert list(d.u[:, 0]) == g["u1"] and list(d.vhat[:, 0]) == g["vhat1"]
            assert list(d.r[:, 0]) == g["r1"]


def test_zero_column_stays_zero():
    N = 16
    x = np.zeros((N, 1))
    d = ko.decompose(x, ko.sign_mask(0, N), 3)
    assert not d.u.any() and not d.vhat.any() and not d.r.any()
    q = ko.quantise(x, 0, 3)
    assert not q.codes_u.any() and not q.codes_v.any()


def test_zero_inputs_keep_sign_zero():
    """sign(0) = 0 (the paper leaves it open): an exact zero entry is left untouched by the
    two Q_N steps of the first block."""
    x = _gauss(64, 1, seed=9)
    x[[3, 17, 40]] = 0.0
    d = ko.decompose(x, ko.sign_mask(2, 64), 1, P=lambda z: np.zeros_like(z))
    assert d.u[3, 0] == 0.0 and d.u[17, 0] == 0.0 and d.u[40, 0] == 0.0


# ---------------------------------------------------------------------------
# Tie-follow protocol (test machinery for the discontinuous sign)
# ---------------------------------------------------------------------------


def test_tie_follow_counts():
    N, k = 64, 2
    x = _gauss(N, 2, seed=4)
    eps = ko.sign_mask(4, N)
    ref = ko.decompose(x, eps, k)
    # rebuild the oracle's own decisions, then plant disagreements
    own = np.zeros((4 * k, N, 2), dtype=np.int8)
    d0 = ko.decompose(x, eps, k, follow=own, tau_abs=np.full(2, -1.0))  # tau < 0: never follow
    assert d0.ties == 0 and d0.hard_mismatches > 0
    big = ko.decompose(x, eps, k, follow=own, tau_abs=np.full(2, 1e9))   # follow everything
    assert big.ties == 4 * k * N * 2 and big.hard_mismatches == 0
    np.testing.assert_array_equal(big.u, 0.0)
    assert np.isfinite(ref.u).all()


# ---------------------------------------------------------------------------
# Codes and packing
# ---------------------------------------------------------------------------


def test_codes_boundaries_exhaustive():
    c1, c2 = np.float32(0.75), np.float32(0.25)
    cent = ko.centres(np.array([c1], np.float64), np.array([c2], np.float64))
    m = np.float32(0.75)
    vals = []
    expect = []
    for b, lo in ((-m, 0), (np.float32(0.0), 1), (m, 2)):
        below = np.nextafter(b, np.float32(-np.inf))
        above = np.nextafter(b, np.float32(np.inf))
        vals += [below, b, above]
        expect += [lo, lo, lo + 1]                 # ties go to the lower code
    vals += [np.float32(-5), np.float32(5)]
    expect += [0, 3]
    got = ko.codes(np.array(vals, dtype=np.float32)[:, None], cent)[:, 0]
    np.testing.assert_array_equal(got, expect)


def test_codes_c2_larger_than_c1():
    cent = ko.centres(np.array([0.25]), np.array([0.75]))
    np.testing.assert_allclose(cent[0], [-1.0, -0.5, 0.5, 1.0])
    got = ko.codes(np.array([[-0.76], [-0.74], [0.1], [0.74], [0.76]]), cent)[:, 0]
    np.testing.assert_array_equal(got, [0, 1, 2, 2, 3])


def test_pack_layout_and_roundtrip():
    code = np.zeros((33, 2), dtype=np.int64)
    code[0, 0] = 3
    code[17, 0] = 2
    code[32, 1] = 1
    w = ko.pack_codes(code)
    assert w.shape == (2, 3)
    assert w[0, 0] == 3 and w[0, 1] == (2 << 2) and w[0, 2] == 0
    assert w[1, 2] == 1
    rng = np.random.default_rng(1)
    c = rng.integers(0, 4, size=(100, 7))
    np.testing.assert_array_equal(ko.unpack_codes(ko.pack_codes(c), 100), c)


def test_bits_per_weight_accounting():
    """App. C: 4NM code bits + 4 fp16 magnitudes per column = 4 + 64/N bits/weight."""
    N, M = 4096, 11008
    code_bits = 2 * 2 * N * M
    meta_bits = 4 * 16 * M
    assert (code_bits + meta_bits) / (N * M) == pytest.approx(4 + 64 / N)


def test_reconstruct_n2():
    eps = np.array([1.0, -1.0])
    cu = np.array([[-2.0, -1.0, 1.0, 2.0]])
    cv = np.array([[-4.0, -3.0, 3.0, 4.0]])
    code_u = np.array([[3], [0]])
    code_v = np.array([[1], [2]])
    W = ko.reconstruct(code_u, code_v, cu, cv, eps)
    # U_q = (2, -2); V_q = (-3, 3); P = swap -> P V_q = (3, -3)
    np.testing.assert_allclose(W[:, 0], [5.0, -5.0], atol=1e-14)


def test_follow_floor_gates_following():
    """Below the follow floor the oracle takes its own signs and counts nothing."""
    N, k = 64, 3
    x = _gauss(N, 2, seed=6)
    eps = ko.sign_mask(6, N)
    ref = ko.decompose(x, eps, k)
    planted = np.zeros((4 * k, N, 2), dtype=np.int8)          # a device that always says 0
    gated = ko.decompose(x, eps, k, follow=planted, tau_abs=np.full(2, 1e9), follow_floor=np.full(2, 1e9))
    assert gated.ties == 0 and gated.hard_mismatches == 0
    np.testing.assert_array_equal(gated.u, ref.u)
    open_gate = ko.decompose(x, eps, k, follow=planted, tau_abs=np.full(2, 1e9), follow_floor=np.zeros(2))
    assert open_gate.ties == 4 * k * N * 2


# ---------------------------------------------------------------------------
# k-means refinement (Sec. 2.1)
# ---------------------------------------------------------------------------


def test_kmeans_hand_worked():
    """values -5,-4 | -1 | 0.5, 1.5 | 6 with centres (-4, -1, 1, 4): one Lloyd step
    gives means -4.5, -1, 1, 6 (assignment by the midpoints -2.5, 0, 2.5)."""
    vals = np.array([-5.0, -4.0, -1.0, 0.5, 1.5, 6.0])[:, None]
    cent = np.array([[-4.0, -1.0, 1.0, 4.0]])
    c1, code, _, _ = ko.kmeans_refine(vals, cent, 1)
    np.testing.assert_array_equal(c1[0], [-4.5, -1.0, 1.0, 6.0])
    np.testing.assert_array_equal(code[:, 0], [0, 0, 1, 2, 2, 3])


def test_kmeans_empty_cluster_keeps_centre_and_order():
    vals = np.array([0.1, 0.2, 0.3])[:, None]
    cent = np.array([[-3.0, -1.0, 1.0, 3.0]])
    c1, _, _, _ = ko.kmeans_refine(vals, cent, 2)
    np.testing.assert_allclose(c1[0], [-3.0, -1.0, 0.2, 3.0])
    assert np.all(np.diff(c1[0]) > 0)


def _sse(vals, cent):
    code = ko.codes(vals, cent)
    return ((vals - ko.dequantise(code, cent)) ** 2).sum(axis=0)


def test_kmeans_sse_non_increasing_and_zero_iters():
    """Lloyd steps never increase the within-cluster squared error; zero iterations
    leave the closed-form centres (Sec. 2.1) untouched."""
    N = 256
    x = _gauss(N, 6, seed=12)
    q0 = ko.quantise(x, 3, 4)
    prev = _sse(q0.dec.u, q0.centres_u)
    for k in (1, 2, 3, 6):
        c, _, _, _ = ko.kmeans_refine(q0.dec.u, q0.centres_u, k)
        cur = _sse(q0.dec.u, c)
        assert np.all(cur <= prev * (1 + 1e-12))
        prev = cur
    c0, code0, _, _ = ko.kmeans_refine(q0.dec.u, q0.centres_u, 0)
    np.testing.assert_array_equal(c0, q0.centres_u)
    np.testing.assert_array_equal(code0, q0.codes_u)
    q3 = ko.quantise(x, 3, 4, kmeans_iters=3)
    assert np.all(_sse(q3.dec.u, q3.centres_u) <= _sse(q0.dec.u, q0.centres_u))


# ---------------------------------------------------------------------------
# Algorithm 2 (App. B): the original vector greedy algorithm
# ---------------------------------------------------------------------------

def test_alg2_hand_worked_n2_swap():
    """N = 2 with the exact swap P (eps = (+1, -1)) and x = (3, 1): ||x||_1 = ||P x||_1,
    so both updates take the vhat branch.  First: P x = (1, 3), s = (1, 1),
    coefficient 4/2 = 2, vhat = (2, 2), r = x - P (2, 2) = (1, -1).  Second:
    P r = (-1, 1), s = (-1, 1), coefficient 2/2 = 1, vhat = (1, 3), r = 0."""
    swap = lambda z: np.asarray(z, dtype=np.float64)[::-1].copy()
    g = ko.greedy_original(np.array([3.0, 1.0]), swap, tol=1e-300, max_updates=8)
    np.testing.assert_array_equal(g.branch, [1, 1])
    np.testing.assert_array_equal(g.coeffs, [2.0, 1.0])
    np.testing.assert_array_equal(g.vhat, [1.0, 3.0])
    np.testing.assert_array_equal(g.u, [0.0, 0.0])
    np.testing.assert_array_equal(g.r, [0.0, 0.0])
    np.testing.assert_array_equal(g.norms, [np.sqrt(10.0), np.sqrt(2.0), 0.0])


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_alg2_prefix_replay_branch_and_drop(seed):
    """Replaying Algorithm 2 for t updates gives the residual r_t entering update t.
    Update t must take the branch with the larger l1 norm of r_t and P r_t, and, with
    no zero entries, lower ||r||^2 by exactly max(||r_t||_1, ||P r_t||_1)^2 / N (the
    squared length of the projection onto the chosen sign vector); the factors must
    reconstruct x exactly."""
    N = 64
    x = _gauss(N, 1, seed=40 + seed)[:, 0]
    eps = ko.sign_mask(seed, N)
    P = ko.POperator(N, eps)
    T = 12
    full = ko.greedy_original(x, P, tol=0.0, max_updates=T)
    assert len(full.branch) == T
    for t in range(T):
        r_t = ko.greedy_original(x, P, tol=0.0, max_updates=t).r
        l1_u, l1_v = np.abs(r_t).sum(), np.abs(P(r_t)).sum()
        assert full.branch[t] == (0 if l1_u > l1_v else 1)
        drop = full.norms[t] ** 2 - full.norms[t + 1] ** 2
        np.testing.assert_allclose(drop, max(l1_u, l1_v) ** 2 / N, rtol=1e-9)
    np.testing.assert_allclose(full.u + P(full.vhat) + full.r, x, atol=1e-12)
    assert np.all(np.diff(full.norms) < 0)


# ---------------------------------------------------------------------------
# Randomized-Hadamard rotation (Sec. 4, Kashin-DCT+H)
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("b", [1, 2, 4, 16, 256, 1024])
def test_hadamard_matches_scipy_sylvester(b):
    scipy_linalg = pytest.importorskip("scipy.linalg")
    np.testing.assert_array_equal(ko.hadamard_matrix(b), scipy_linalg.hadamard(b))


def test_hadamard_orthogonal_brute_force():
    for b in (2, 8, 64):
        H = ko.hadamard_matrix(b)
        np.testing.assert_array_equal(H @ H.T, b * np.eye(b))


def test_rht_block_lengths():
    assert [ko.rht_block(n) for n in (16, 256, 768, 3072, 4096, 11008, 14336, 16384, 32768, 40)] == \
        [16, 256, 256, 1024, 4096, 256, 2048, 16384, 16384, 8]


def test_rht_n2_hand_worked():
    """n = 2, b = 2: y = [[1, 1], [1, -1]] / sqrt 2 applied to (s0 x0, s1 x1), signs
    first (the sign set comes from the SplitMix64 sequence pinned above).  For
    x = (3, 1): y = (3 s0 + s1, 3 s0 - s1) / sqrt 2; the inverse maps it back."""
    for seed in range(8):
        s0, s1 = ko.sign_mask(seed, 2)
        y = ko.randomized_hadamard(np.array([3.0, 1.0]), seed)
        np.testing.assert_allclose(y, np.array([3 * s0 + s1, 3 * s0 - s1]) / np.sqrt(2.0), rtol=0, atol=1e-15)
        np.testing.assert_allclose(ko.randomized_hadamard(y, seed, inverse=True), [3.0, 1.0], rtol=0, atol=1e-15)
    # both sign orders occur among these seeds, so the order of flip and transform is exercised
    assert len({tuple(ko.sign_mask(sd, 2)) for sd in range(8)}) >= 3


def test_rht_spike_is_flat_and_blocks_independent():
    """A unit spike at j spreads to +-1/sqrt(b) over j's block and nowhere else
    (incoherence); the transform acts block by block (n = 768 = 3 blocks of 256)."""
    n, seed = 768, 11
    for j in (0, 300, 767):
        e = np.zeros(n)
        e[j] = 1.0
        y = ko.randomized_hadamard(e, seed)
        blk = j // 256
        inside = y[blk * 256:(blk + 1) * 256]
        np.testing.assert_allclose(np.abs(inside), 1.0 / 16.0, rtol=0, atol=1e-15)
        assert np.count_nonzero(np.delete(y, np.s_[blk * 256:(blk + 1) * 256])) == 0


def test_rht_orthogonal_roundtrip():
    x = _gauss(4096, 3, seed=8)
    y = ko.randomized_hadamard(x, 5)
    np.testing.assert_allclose(np.linalg.norm(y, axis=0), np.linalg.norm(x, axis=0), rtol=1e-13)
    np.testing.assert_allclose(ko.randomized_hadamard(y, 5, inverse=True), x, rtol=0, atol=1e-13)
    # the inverse is the transpose: <R x, z> = <x, R^T z>
    z = _gauss(4096, 3, seed=9)
    np.testing.assert_allclose((y * z).sum(0), (x * ko.randomized_hadamard(z, 5, inverse=True)).sum(0), rtol=1e-12)
