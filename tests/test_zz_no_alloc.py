"""kd_decompose_static: the decomposition for callers that cannot allocate device
memory (its scratch is a static device array inside the library).  Collected last
on purpose; it must pass alone in a fresh process and after the other tests.

Checked through the C ABI: two calls in a row (different vector lengths, so the
shared static tables are rewritten between them) must reproduce kd_decompose with
a caller workspace bit for bit (the same kernels and tables run on both paths), a
repeated call must leave the device's free memory unchanged, a non-finite input
must be reported by kd_read_status_static, and a vector length above the static
limit is refused."""

import ctypes

import numpy as np
import pytest

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def env():
    import torch
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2609_11687_gb300 import build
    build.build()
    from paper_2609_11687_gb300 import kashin as kd
    lib = ctypes.CDLL(kd.LIB_PATH)
    vp, i64 = ctypes.c_void_p, ctypes.c_int64
    lib.kd_decompose_static.argtypes = [vp, ctypes.c_int, ctypes.c_int, i64, i64, i64, ctypes.c_uint64,
                                        ctypes.c_int, ctypes.c_int] + [vp] * 10
    lib.kd_decompose_static.restype = ctypes.c_int
    lib.kd_read_status_static.argtypes = [vp]
    lib.kd_read_status_static.restype = ctypes.c_int
    return torch, kd, lib


def _static(torch, kd, lib, w, iters, seed):
    m, n = w.shape
    words = (n + 15) // 16
    o = {k: torch.empty((m, words), dtype=torch.int32, device="cuda") for k in ("codes_u", "codes_v")}
    for k in ("centres_u", "centres_v", "coeffs"):
        o[k] = torch.empty((m, 4), dtype=torch.float32, device="cuda")
    for k in ("u", "vhat", "resid"):
        o[k] = torch.empty((m, n), dtype=torch.float32, device="cuda")
    st = lib.kd_decompose_static(w.data_ptr(), kd._dtype_code(w.dtype), kd.KD_VEC_ROWS, n, m, w.stride(0),
                                 seed, iters, 0, o["codes_u"].data_ptr(), o["codes_v"].data_ptr(),
                                 o["centres_u"].data_ptr(), o["centres_v"].data_ptr(), o["coeffs"].data_ptr(),
                                 o["u"].data_ptr(), o["vhat"].data_ptr(), o["resid"].data_ptr(), None,
                                 torch.cuda.current_stream().cuda_stream)
    assert st == kd.KD_OK, kd.status_string(st)
    return o


def test_static_scratch_matches_workspace_path(env):
    torch, kd, lib = env
    g = torch.Generator().manual_seed(123)
    cases = [(torch.randn((10, 4096), generator=g) * 0.02).half().cuda(),
             (torch.randn((7, 256), generator=g) * 0.02).cuda()]
    for call, w in enumerate(cases):             # two calls in a row, different n
        seed = 40 + call
        got = _static(torch, kd, lib, w, 16, seed)
        ref = kd.decompose(w, 16, seed, factors=True, coeffs=True)
        torch.cuda.synchronize()
        for k in ("codes_u", "codes_v", "centres_u", "centres_v", "coeffs", "u", "vhat", "resid"):
            assert torch.equal(got[k], getattr(ref, k)), (call, k)
        assert lib.kd_read_status_static(torch.cuda.current_stream().cuda_stream) == kd.KD_OK


def test_static_call_allocates_nothing(env):
    """A repeated call (its kernels already loaded by the first) must not change the
    device's free memory: the scratch is the static array, nothing else is taken."""
    torch, kd, lib = env
    g = torch.Generator().manual_seed(7)
    w = (torch.randn((12, 4096), generator=g) * 0.02).half().cuda()
    first = _static(torch, kd, lib, w, 8, 3)
    torch.cuda.synchronize()
    free_before, _ = torch.cuda.mem_get_info()
    seed, iters = 3, 8
    m, n = w.shape
    st = lib.kd_decompose_static(w.data_ptr(), kd.KD_F16, kd.KD_VEC_ROWS, n, m, n, seed, iters, 0,
                                 first["codes_u"].data_ptr(), first["codes_v"].data_ptr(),
                                 first["centres_u"].data_ptr(), first["centres_v"].data_ptr(),
                                 first["coeffs"].data_ptr(), first["u"].data_ptr(), first["vhat"].data_ptr(),
                                 first["resid"].data_ptr(), None, torch.cuda.current_stream().cuda_stream)
    assert st == kd.KD_OK
    assert lib.kd_read_status_static(torch.cuda.current_stream().cuda_stream) == kd.KD_OK
    torch.cuda.synchronize()
    free_after, _ = torch.cuda.mem_get_info()
    assert free_after == free_before


def test_static_status_reports_nonfinite_input(env):
    """A NaN in the input sets the status word in the static array; the next call with
    finite inputs clears it again."""
    torch, kd, lib = env
    w = (torch.arange(4 * 256, dtype=torch.float32).reshape(4, 256) * 1e-3 - 0.5).cuda()
    bad = w.clone()
    bad[1, 17] = float("nan")
    stream = torch.cuda.current_stream().cuda_stream
    _static(torch, kd, lib, bad, 4, 1)
    assert lib.kd_read_status_static(stream) == kd.KD_ERR_NONFINITE
    _static(torch, kd, lib, w, 4, 1)
    assert lib.kd_read_status_static(stream) == kd.KD_OK


def test_static_scratch_refuses_long_vectors(env):
    torch, kd, lib = env
    w = torch.zeros((2, 11008), dtype=torch.float16, device="cuda")
    dummy = torch.empty(64, dtype=torch.int32, device="cuda")
    st = lib.kd_decompose_static(w.data_ptr(), kd.KD_F16, kd.KD_VEC_ROWS, 11008, 2, 11008, 0, 4, 0,
                                 dummy.data_ptr(), dummy.data_ptr(), dummy.data_ptr(), dummy.data_ptr(),
                                 None, None, None, None, None, None)
    assert st == kd.KD_ERR_WORKSPACE
