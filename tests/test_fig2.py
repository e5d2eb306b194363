"""Fig. 2 on the CPU: the original greedy algorithm (Algorithm 2) against
Algorithm 1 on a Gaussian vector, summarised by the per-update residual decay
and by the four-level quantiser distortion of each factor (oracle/fig2.py).

The distortion measure is pinned first to textbook values: 0.1175 for a
Gaussian (the Lloyd-Max optimum for four levels, Max 1960) and 1/16 for a
uniform density (four equal cells, each contributing width^2 / 12)."""

import numpy as np
import pytest

from oracle import fig2
from paper_2609_11687_gb300 import synth


def test_distortion_gaussian_is_lloyd_max():
    z = np.random.default_rng(5).standard_normal(200_000)
    assert abs(fig2.four_level_distortion(z) - 0.1175) < 0.002


def test_distortion_uniform_is_one_sixteenth():
    z = np.random.default_rng(6).uniform(-1.0, 1.0, 200_000)
    assert abs(fig2.four_level_distortion(z) - 1.0 / 16.0) < 0.001


def test_distortion_four_spikes_is_zero():
    z = np.repeat([-3.0, -1.0, 1.0, 3.0], 50)
    assert fig2.four_level_distortion(z) < 1e-20


@pytest.fixture(scope="module")
def fig2_run():
    x = synth.generate(synth.gaussian_vectors(2000, 1, seed=0))[0].double().numpy()
    return fig2.reproduce(x)


def test_fig2_convergence_rates_comparable(fig2_run):
    """Fig. 2 left: Algorithm 1 converges at nearly the original algorithm's rate.
    Over 64 updates its log-decay is at least 3/4 of Algorithm 2's."""
    r = fig2_run
    assert r["updates"] == 64
    assert np.log(r["rate_alg1"]) <= 0.75 * np.log(r["rate_alg2"])
    assert np.all(np.diff(r["norms_alg1"]) < 0)


def test_fig2_alg1_factors_have_four_peaks(fig2_run):
    """Fig. 2 centre/right: Algorithm 1's factors concentrate on four peaks; their
    best four-level distortion is far below a Gaussian's 0.1175 (the input's own)."""
    d = fig2_run["distortion"]
    assert d["input"] > 0.1
    assert d["alg1_u"] < 0.03 and d["alg1_vhat"] < 0.03


def test_fig2_closed_form_centres_near_lloyd_optimum(fig2_run):
    """Sec. 2.1: the closed-form centres +-c1 +-c2 (+-d1 +-d2) sit where Lloyd's
    algorithm ends: within 3 % of the outer centre."""
    r = fig2_run
    for cf, opt in ((r["closed_form_u"], r["optimal_u"]), (r["closed_form_v"], r["optimal_v"])):
        assert np.abs(cf - opt).max() <= 0.03 * cf[3]
