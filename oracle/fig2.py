"""Fig. 2 reproduction on the CPU (TEST INFRASTRUCTURE, like the rest of oracle/).

Fig. 2 runs one Gaussian vector ``x ~ N(0, I_N)``, ``N = 10^4``, through the
original greedy algorithm (Algorithm 2, App. B) and through Algorithm 1, and
compares (left) the residual norm against the number of greedy updates and
(centre, right) the empirical densities of the two factors at convergence.
The paper reports that Algorithm 1 converges at nearly the original's rate and
gives each factor four sharp symmetric peaks.

This module computes the same quantities with the fp64 oracle and sums up the
densities by one number: the distortion of the best four-level (1-D, 4-centre
k-means) quantiser of a factor, divided by the factor's variance.  Four sharp
peaks give a value near zero; a Gaussian gives 0.1175 (the Lloyd-Max optimum
for four levels, Max 1960); a uniform density gives 1/16.

Run ``python -m oracle.fig2 [N]`` for the text summary at N (default 10^4).
"""

from __future__ import annotations

import sys

import numpy as np

from oracle import kashin_oracle as ko


def four_level_distortion(values: np.ndarray, init: np.ndarray | None = None, iters: int = 100) -> float:
    """min over starting points of the 4-centre Lloyd distortion / variance.

    Starts from the 1/8, 3/8, 5/8, 7/8 quantiles and, if given, from ``init``
    (e.g. the closed-form centres); ``iters`` Lloyd iterations from each.
    """
    v = np.asarray(values, dtype=np.float64).reshape(-1, 1)
    starts = [np.quantile(v[:, 0], [0.125, 0.375, 0.625, 0.875])]
    if init is not None:
        starts.append(np.sort(np.asarray(init, dtype=np.float64)))
    best = np.inf
    for c0 in starts:
        c, code, _, _ = ko.kmeans_refine(v, c0[None, :], iters)
        d = float(((v[:, 0] - c[0][code[:, 0]]) ** 2).mean())
        best = min(best, d)
    return best / float(v.var())


def optimal_centres(values: np.ndarray, init: np.ndarray, iters: int = 100) -> np.ndarray:
    """Lloyd-converged four centres started from ``init``."""
    v = np.asarray(values, dtype=np.float64).reshape(-1, 1)
    c, _, _, _ = ko.kmeans_refine(v, np.sort(np.asarray(init, dtype=np.float64))[None, :], iters)
    return c[0]


def reproduce(x: np.ndarray, sign_seed: int = 1, blocks: int = 16) -> dict:
    """Both algorithms on ``x`` with the same operator P; equal numbers of updates
    (4 per block of Algorithm 1)."""
    x = np.asarray(x, dtype=np.float64)
    n = x.shape[0]
    eps = ko.sign_mask(sign_seed, n)
    P = ko.POperator(n, eps)
    a1 = ko.decompose(x[:, None], eps, blocks, P=P)
    a2 = ko.greedy_original(x, P, tol=0.0, max_updates=4 * blocks)
    cu = ko.centres(a1.coeffs[0], a1.coeffs[1])[0]
    cv = ko.centres(a1.coeffs[2], a1.coeffs[3])[0]
    norms1 = a1.step_norms[:, 0]
    norms2 = a2.norms
    updates = len(norms2) - 1

    def rate(norms, k):
        return float(np.exp(np.log(norms[k] / norms[0]) / k))

    return {
        "n": n,
        "updates": updates,
        "norms_alg1": norms1,
        "norms_alg2": norms2,
        "branch_alg2": a2.branch,
        # geometric per-update decay of ||r|| over the first `updates` updates
        "rate_alg1": rate(norms1, updates),
        "rate_alg2": rate(norms2, updates),
        "closed_form_u": cu,
        "closed_form_v": cv,
        "optimal_u": optimal_centres(a1.u[:, 0], cu),
        "optimal_v": optimal_centres(a1.vhat[:, 0], cv),
        "distortion": {
            "alg1_u": four_level_distortion(a1.u[:, 0], cu),
            "alg1_vhat": four_level_distortion(a1.vhat[:, 0], cv),
            "alg2_u": four_level_distortion(a2.u),
            "alg2_vhat": four_level_distortion(a2.vhat),
            "input": four_level_distortion(x),
        },
        "factors": {"alg1_u": a1.u[:, 0], "alg1_vhat": a1.vhat[:, 0], "alg2_u": a2.u, "alg2_vhat": a2.vhat},
    }


def main(argv=None) -> None:
    argv = sys.argv[1:] if argv is None else argv
    n = int(argv[0]) if argv else 10_000
    from paper_2609_11687_gb300 import synth
    x = synth.generate(synth.gaussian_vectors(n, 1, seed=0))[0].double().numpy()
    res = reproduce(x)
    print(f"N = {n}, {res['updates']} greedy updates each (Algorithm 1: 16 blocks)")
    print("residual ||r|| every 4 updates:")
    for k in range(0, res["updates"] + 1, 4):
        print(f"  {k:3d}  alg1 {res['norms_alg1'][k]:.4e}  alg2 {res['norms_alg2'][k]:.4e}")
    print(f"per-update decay: alg1 {res['rate_alg1']:.4f}  alg2 {res['rate_alg2']:.4f}")
    print("alg2 branches (0 = u, 1 = vhat):", "".join(map(str, res["branch_alg2"].tolist())))
    for k, v in res["distortion"].items():
        print(f"four-level distortion / variance  {k:10s} {v:.4f}")
    print("closed-form u centres", np.round(res["closed_form_u"], 4), " Lloyd-optimal", np.round(res["optimal_u"], 4))
    print("closed-form v centres", np.round(res["closed_form_v"], 4), " Lloyd-optimal", np.round(res["optimal_v"], 4))
    for name, f in res["factors"].items():
        h, e = np.histogram(f, bins=24)
        print(f"histogram {name:10s} [{e[0]:+.3f}, {e[-1]:+.3f}]:", " ".join(str(int(c)) for c in h))


if __name__ == "__main__":
    main()
