"""Parity harness: compare device results with the CPU oracle on the same inputs.

Tolerances (from the stated contract, per vector):
  u, vhat      ||gpu - ora||_inf / ||ora||_inf <= 1e-5
  coefficients |gpu - ora| / ora <= 1e-5 ; centres relative to their outer value
  codes        identical, except entries whose oracle value lies within
               1e-6 * (a1 + a2) of a decision boundary; those <= 0.01 % of entries
  x = u + P vhat + r  from the device factors: relative l2 error <= 1e-6
  ||r_k||_2    per vector, device against oracle: within RESID_REL (relative) where
               the oracle's residual is above R_RESOLVED * ||x||, at most RESID_RATIO
               times the oracle's above the fp32 floor, and below RESID_FLOOR * ||x||
               under it (there the oracle no longer follows the device's signs and the
               two trajectories, each still shrinking, drift apart by up to ~10x).
               The residual falls by about 5-8x per block, so a kernel that stopped
               early or went wrong in a late block fails: measured on the 7B layer's
               n = 4096 and 11008 matrices, 2.7e-4 relative at k = 8, at most 2e-9
               ||x|| at k = 16, against 2e-6 ||x|| for a run stopped after 8 of 16
               blocks.
  E            E = ||W - W_hat||_F / ||W||_F of the dequantised weight (App. C), device
               (kd_reconstruct on its codes and centres) against the oracle's (its own
               centres and codes, fp64, taking the device's code only inside the 1e-6
               boundary window, where either code is allowed): |E_gpu - E_ora| <= 1e-6
               E_ora (measured 1-2e-7 where no code differs).
Signs: Alg. 1 takes sign() of every entry at every step; where fp32 and fp64
disagree on a value within rounding of zero the trajectories would split, so
the oracle follows the device's recorded sign wherever its own argument is
within tau_abs = TAU * ||x||_inf of zero (fp32 rounding error scales with the
largest magnitude the vector carries, which heavy-tailed and outlier inputs make
much larger than its rms) and counts any other disagreement as a hard failure
(must be zero).  Below the device's rounding floor (residual
norm < FLOOR * 2^-24 * ||x||_2) fp32 cannot resolve the residual at all, so the
oracle stops following there and takes its own signs; those steps change u and
vhat by at most ||rho||_2 / sqrt(N) each (Eq. lambda_bound), which the 1e-5
factor tolerance absorbs.
"""

from __future__ import annotations

import dataclasses

import numpy as np

from oracle import kashin_oracle as ko

TAU = 1e-5          # tie window, relative to the vector's max |x_i|
FLOOR = 16.0        # follow only while ||rho||_2 >= FLOOR * 2^-24 * ||x||_2
TOL_FACTOR = 1e-5   # u, vhat, coefficients, centres
TOL_RECON = 1e-6    # x = u + P vhat + r from device factors
CODE_WINDOW = 1e-6  # near-boundary window, relative to a1 + a2
CODE_FRAC = 1e-4    # at most 0.01 % of entries may differ, all inside the window
R_RESOLVED = 1e-5   # residual norms compared where the oracle's ||r_k|| / ||x|| is at least this ...
RESID_REL = 2e-3    # ... to this relative difference
RESID_RATIO = 2.0   # every vector: r_gpu <= max(RESID_RATIO * r_ora, RESID_FLOOR) ...
RESID_FLOOR = 1e-7  # ... with ||r_k|| / ||x|| measured relative to ||x||: the fp32 floor
TOL_E = 1e-6        # |E_gpu - E_ora| <= TOL_E * E_ora, E = ||W - W_hat||_F / ||W||_F


@dataclasses.dataclass
class ParityReport:
    n: int
    m: int
    hard: int
    ties: int
    tie_flips: int
    u_err: float
    v_err: float
    coef_err: float
    cent_err: float
    code_diff: int
    code_diff_outside: int
    code_near: int
    recon_err: float
    entries: int
    # per-vector residual norms ||r_k||_2 / ||x||_2 (device, oracle) and the
    # reconstruction-error contract E = ||W - W_hat||_F / ||W||_F (when measured)
    r_gpu: np.ndarray = dataclasses.field(default=None, repr=False)
    r_ora: np.ndarray = dataclasses.field(default=None, repr=False)
    resid_err: float = 0.0
    resid_ratio: float = 0.0
    e_gpu: float = float("nan")
    e_ora: float = float("nan")
    e_ora_own: float = float("nan")

    def check(self, code_budget: bool = True):
        """code_budget=False for degenerate inputs (constant vectors, single spikes)
        whose values sit on a decision boundary by construction: every mismatch
        must still lie inside the boundary window."""
        assert self.hard == 0, f"{self.hard} sign decisions disagree outside the tie window"
        assert self.u_err <= TOL_FACTOR, f"u max rel err {self.u_err:.3e}"
        assert self.v_err <= TOL_FACTOR, f"vhat max rel err {self.v_err:.3e}"
        assert self.coef_err <= TOL_FACTOR, f"coefficient rel err {self.coef_err:.3e}"
        assert self.cent_err <= TOL_FACTOR, f"centre rel err {self.cent_err:.3e}"
        assert self.code_diff_outside == 0, f"{self.code_diff_outside} code mismatches away from a boundary"
        if code_budget:
            assert self.code_diff <= CODE_FRAC * self.entries, f"{self.code_diff} code mismatches"
        assert self.recon_err <= TOL_RECON, f"x = u + P vhat + r rel err {self.recon_err:.3e}"
        check_residuals(self.r_gpu, self.r_ora)
        if not np.isnan(self.e_gpu):
            assert abs(self.e_gpu - self.e_ora) <= TOL_E * self.e_ora, \
                f"reconstruction error E: device {self.e_gpu:.9f} oracle {self.e_ora:.9f}"


def check_residuals(r_gpu: np.ndarray, r_ora: np.ndarray):
    """Residual norms ||r_k|| / ||x|| per vector, device against oracle (Alg. 1's
    residual after k blocks): close where the oracle's is resolved in fp32, at most
    RESID_RATIO times the oracle's above the fp32 floor, under the floor below it."""
    err, _ = residual_stats(r_gpu, r_ora)
    assert err <= RESID_REL, f"residual norm differs by {err:.3e} relative where resolved"
    bad = np.flatnonzero(r_gpu > np.maximum(RESID_RATIO * r_ora, RESID_FLOOR))
    assert bad.size == 0, (f"{bad.size} vectors with a residual norm above max({RESID_RATIO} x oracle, "
                           f"{RESID_FLOOR:g}): e.g. vector {bad[0]} device {r_gpu[bad[0]]:.3e} "
                           f"oracle {r_ora[bad[0]]:.3e}")


def _rel_inf(a, b):
    """max over columns of ||a-b||_inf / ||b||_inf (columns with b == 0 use abs error)."""
    num = np.abs(a - b).max(axis=0)
    den = np.abs(b).max(axis=0)
    out = np.where(den > 0, num / np.where(den > 0, den, 1), num)
    return float(out.max()) if out.size else 0.0


def compare(x: np.ndarray, seed: int, iters: int, dev: dict, P_oracle=None, kmeans_iters: int = 0) -> ParityReport:
    """x: (N, M) float64 inputs (exact values the device saw).  dev: numpy arrays
    from the device, vector-major: u, vhat, resid (M, N) float32, coeffs (M, 4),
    centres_u/centres_v (M, 4), codes_u/codes_v (M, N) int, trace (M, 4k, N) int8."""
    N, M = x.shape
    eps = ko.sign_mask(seed, N)
    P = P_oracle if P_oracle is not None else ko.POperator(N, eps)
    xmax = np.abs(x).max(axis=0)
    trace = np.transpose(dev["trace"], (1, 2, 0)).astype(np.int8)    # (4k + 2 kmeans, N, M)
    follow = trace[:4 * iters]
    floor = FLOOR * 2.0 ** -24 * np.linalg.norm(x, axis=0)
    d = ko.decompose(x, eps, iters, follow=follow, tau_abs=TAU * xmax, P=P, follow_floor=floor)
    cu = ko.centres(d.coeffs[0], d.coeffs[1])
    cv = ko.centres(d.coeffs[2], d.coeffs[3])
    km_hard = 0
    if kmeans_iters > 0:
        # Lloyd refinement (Sec. 2.1) following the device's assignment near a boundary
        km = trace[4 * iters:].reshape(kmeans_iters, 2, N, M)
        wu = CODE_WINDOW * np.abs(cu[:, 3])
        wv = CODE_WINDOW * np.abs(cv[:, 3])
        cu, code_u, _, h1 = ko.kmeans_refine(d.u, cu, kmeans_iters, follow=km[:, 0], window=wu)
        cv, code_v, _, h2 = ko.kmeans_refine(d.vhat, cv, kmeans_iters, follow=km[:, 1], window=wv)
        km_hard = h1 + h2
    else:
        code_u = ko.codes(d.u, cu)
        code_v = ko.codes(d.vhat, cv)

    u_g = dev["u"].T.astype(np.float64)
    v_g = dev["vhat"].T.astype(np.float64)
    r_g = dev["resid"].T.astype(np.float64)
    u_err = _rel_inf(u_g, d.u)
    v_err = _rel_inf(v_g, d.vhat)
    co_g = dev["coeffs"].T.astype(np.float64)
    den = np.where(d.coeffs != 0, np.abs(d.coeffs), 1.0)
    coef_err = float((np.abs(co_g - d.coeffs) / den).max()) if M else 0.0
    cent_err = 0.0
    for cg, co in ((dev["centres_u"], cu), (dev["centres_v"], cv)):
        outer = np.abs(co[:, 3])
        dd = np.abs(cg.astype(np.float64) - co).max(axis=1)
        cent_err = max(cent_err, float(np.where(outer > 0, dd / np.where(outer > 0, outer, 1), dd).max()))

    diff = 0
    outside = 0
    near_total = 0
    followed = []   # oracle codes, taking the device's inside the boundary window
    for cg, co, vals, cent in ((dev["codes_u"], code_u, d.u, cu), (dev["codes_v"], code_v, d.vhat, cv)):
        cg = cg.T
        mism = cg != co
        dist = ko.boundary_distance(vals, cent)
        window = CODE_WINDOW * np.abs(cent[:, 3])[None, :]
        near = dist <= window
        near_total += int(near.sum())
        diff += int(mism.sum())
        outside += int((mism & ~near).sum())
        followed.append(np.where(near, cg, co))

    Pv = P(v_g)
    nx = np.linalg.norm(x, axis=0)
    nx1 = np.where(nx > 0, nx, 1)
    recon = np.linalg.norm(x - u_g - Pv - r_g, axis=0) / nx1
    r_gpu = np.linalg.norm(r_g, axis=0) / nx1
    r_ora = np.linalg.norm(d.r, axis=0) / nx1
    resid_err, resid_ratio = residual_stats(r_gpu, r_ora)
    e_gpu = e_ora = e_ora_own = float("nan")
    if "w_hat" in dev:
        # App. C: the dequantised weight W_hat = U_q + P V_q; device from kd_reconstruct on
        # its own codes and centres, oracle from its own centres and codes (fp64, dense
        # P).  The allowed near-boundary code differences each move E by up to about
        # 1e-5 / sqrt(entries) (the two candidate centres are equally far from the
        # factor entry, not from the weight), so the contract compares with the oracle's
        # codes following the device's inside the boundary window; the oracle's own
        # codes give e_ora_own, reported beside it.
        nW = np.linalg.norm(x)
        e_gpu = float(np.linalg.norm(x - dev["w_hat"].T.astype(np.float64)) / nW)
        wh_ora = ko.dequantise(followed[0], cu) + P(ko.dequantise(followed[1], cv))
        e_ora = float(np.linalg.norm(x - wh_ora) / nW)
        wh_own = ko.dequantise(code_u, cu) + P(ko.dequantise(code_v, cv))
        e_ora_own = float(np.linalg.norm(x - wh_own) / nW)
    return ParityReport(n=N, m=M, hard=d.hard_mismatches + km_hard, ties=d.ties, tie_flips=d.tie_flips, u_err=u_err,
                        v_err=v_err, coef_err=coef_err, cent_err=cent_err, code_diff=diff,
                        code_diff_outside=outside, code_near=near_total, recon_err=float(recon.max()),
                        entries=2 * N * M, r_gpu=r_gpu, r_ora=r_ora, resid_err=resid_err,
                        resid_ratio=resid_ratio, e_gpu=e_gpu, e_ora=e_ora, e_ora_own=e_ora_own)


def residual_stats(r_gpu: np.ndarray, r_ora: np.ndarray):
    """Per-vector residual norms (relative to ||x||), device against oracle.
    Returns (largest relative disagreement among vectors whose oracle residual is
    resolved in fp32, largest ratio r_gpu / r_ora over all vectors with r_ora > 0)."""
    res = r_ora >= R_RESOLVED
    err = float((np.abs(r_gpu[res] - r_ora[res]) / r_ora[res]).max()) if res.any() else 0.0
    pos = r_ora > 0
    ratio = float((r_gpu[pos] / r_ora[pos]).max()) if pos.any() else 0.0
    return err, ratio


def device_outputs(kd, w_dev, iters, seed, trace=True, layout="rows", kmeans_iters=0, w_hat=False):
    """Run kd_decompose with every optional output and return numpy arrays; with
    w_hat, also kd_reconstruct's fp32 W_hat from the device's codes and centres."""
    out = kd.decompose(w_dev, iters, seed, layout=layout, factors=True, coeffs=True, trace=trace,
                       kmeans_iters=kmeans_iters)
    n = out.u.shape[1]
    import torch
    wh = kd.reconstruct(out, n, seed, dtype=torch.float32) if w_hat else None
    torch.cuda.synchronize()
    res = {
        "u": out.u.cpu().numpy(), "vhat": out.vhat.cpu().numpy(), "resid": out.resid.cpu().numpy(),
        "coeffs": out.coeffs.cpu().numpy(), "centres_u": out.centres_u.cpu().numpy(),
        "centres_v": out.centres_v.cpu().numpy(),
        "codes_u": kd.unpack_codes(out.codes_u, n), "codes_v": kd.unpack_codes(out.codes_v, n),
        "words_u": out.codes_u.cpu().numpy(), "words_v": out.codes_v.cpu().numpy(),
    }
    if trace:
        res["trace"] = out.trace.cpu().numpy()
    if wh is not None:
        res["w_hat"] = wh.cpu().numpy()
    return res
