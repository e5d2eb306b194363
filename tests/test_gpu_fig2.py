"""Fig. 2's properties on the device path: Gaussian vectors at the figure's own
N = 10^4 (2^4 5^4, the run-time-length path) and at the compiled lengths around
it (8192, 11008, 16384).
Algorithm 1 on the GPU must leave both factors on four sharp peaks (best
four-level distortion far below a Gaussian's 0.1175), and the device's k-means
refinement must converge to the Lloyd optimum near the closed-form centres."""

import numpy as np
import pytest

from oracle import fig2
from paper_2609_11687_gb300 import synth

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


@pytest.mark.parametrize("n", [8192, 10000, 11008, 16384])
def test_gpu_fig2_four_peaks_and_lloyd(kd, n):
    import torch
    m = 4
    w = synth.generate(synth.gaussian_vectors(n, m, seed=n), device="cuda")
    closed = kd.decompose(w, ITERS, 1, factors=True)
    refined = kd.decompose(w, ITERS, 1, kmeans_iters=30)
    torch.cuda.synchronize()
    u = closed.u.double().cpu().numpy()
    vh = closed.vhat.double().cpu().numpy()
    cu = closed.centres_u.double().cpu().numpy()
    cv = closed.centres_v.double().cpu().numpy()
    ru = refined.centres_u.double().cpu().numpy()
    rv = refined.centres_v.double().cpu().numpy()
    for j in range(m):
        assert fig2.four_level_distortion(u[j], cu[j]) < 0.03
        assert fig2.four_level_distortion(vh[j], cv[j]) < 0.03
        # device Lloyd result = oracle Lloyd result from the same start, on the device factors
        np.testing.assert_allclose(ru[j], fig2.optimal_centres(u[j], cu[j], iters=30), rtol=0, atol=1e-3 * cu[j, 3])
        np.testing.assert_allclose(rv[j], fig2.optimal_centres(vh[j], cv[j], iters=30), rtol=0, atol=1e-3 * cv[j, 3])
        # the closed form already sits near that optimum (Sec. 2.1)
        assert np.abs(ru[j] - cu[j]).max() <= 0.03 * cu[j, 3]
        assert np.abs(rv[j] - cv[j]).max() <= 0.03 * cv[j, 3]
