"""C-ABI checks that need no GPU: the library builds/loads, exports every entry
point include/kashin.h declares, and its host-only logic (sign mask, plan
lookup, workspace sizing, argument validation) behaves.  No kernel is launched."""

import ctypes
import os
import re

import numpy as np
import pytest

from oracle import kashin_oracle as ko

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "kashin.h")


@pytest.fixture(scope="module")
def kd():
    from paper_2609_11687_gb300 import build
    build.build()
    from paper_2609_11687_gb300 import kashin
    return kashin


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(kd_[a-z_]+)\s*\(", src)))


def test_header_declares_expected_entry_points():
    names = declared_functions()
    for must in ("kd_decompose", "kd_reconstruct", "kd_apply_p", "kd_signs", "kd_workspace_size",
                 "kd_read_status", "kd_supported", "kd_status_string", "kd_version"):
        assert must in names


def test_library_exports_every_declared_symbol(kd):
    lib = ctypes.CDLL(kd.LIB_PATH)
    for name in declared_functions():
        assert hasattr(lib, name), f"{name} declared in kashin.h but not exported"
    assert set(declared_functions()) <= set(kd.EXPORTS)


def test_version_and_status_strings(kd):
    assert "libkashin" in kd.version()
    assert kd.status_string(kd.KD_OK) == "KD_OK"
    assert kd.status_string(kd.KD_ERR_NONFINITE) == "KD_ERR_NONFINITE"
    assert kd.status_string(kd.KD_ERR_TIMEOUT) == "KD_ERR_TIMEOUT"
    assert kd.status_string(99) == "KD_ERR_UNKNOWN"


@pytest.mark.parametrize("seed,n", [(0, 16), (1, 257), (0xDEADBEEFCAFEF00D, 4096), (2**64 - 1, 100)])
def test_kd_signs_match_oracle(kd, seed, n):
    np.testing.assert_array_equal(kd.kd_signs(seed, n), ko.sign_mask(seed, n).astype(np.int8))


TUNED = (16, 32, 64, 128, 256, 512, 768, 1024, 1536, 2048, 3072, 4096, 8192, 11008, 14336, 16384)


def _smooth(n):
    """1 <= n <= 16384 with every prime factor in {2, 3, 5, 7, 11, 13, 43}."""
    if n < 1 or n > 16384:
        return False
    for p in (2, 3, 5, 7, 11, 13, 43):
        while n % p == 0:
            n //= p
    return n == 1


def test_supported_lengths(kd):
    for n in TUNED:
        assert kd.kd_supported(n) == kd.KD_OK and kd.kd_tuned(n)
    # the run-time-length path: every other length whose prime factors are in the set
    for n in (1, 2, 3, 15, 43, 100, 2560, 4095, 5120, 13824, 16000):
        assert kd.kd_supported(n) == kd.KD_OK and not kd.kd_tuned(n)
    for n in (0, -16, 17, 4094, 16385, 32768):
        assert kd.kd_supported(n) == kd.KD_ERR_UNSUPPORTED_N and not kd.kd_tuned(n)


def test_supported_set_is_the_factor_rule(kd):
    got = [n for n in range(0, 16400) if kd.kd_supported(n) == kd.KD_OK]
    assert got == [n for n in range(0, 16400) if _smooth(n)]
    assert [n for n in range(0, 16400) if kd.kd_tuned(n)] == list(TUNED)


def test_workspace_size_register_plans(kd):
    # plans that keep u on chip need only the tables: no device query
    for n in (256, 768, 4096):
        ws = kd.kd_workspace_size(n)
        assert ws >= 256 + 8 * n + n // 8 and ws % 256 == 0   # status, sign bits, pass-0 twiddles
    assert kd.kd_workspace_size(4094) == 0


def test_argument_validation_without_gpu(kd):
    null = None
    # unsupported length
    st = kd.kd_decompose(1, 0, 0, 4094, 4, 4094, 0, 4, 0, 1, 1, 1, 1, null, null, null, null, null, 1, 1 << 20, null)
    assert st == kd.KD_ERR_UNSUPPORTED_N
    # out-of-range refinement count
    assert kd.kd_decompose(1, 0, 0, 256, 4, 256, 0, 4, 65, 1, 1, 1, 1, null, null, null, null, null, 1, 1 << 20,
                           null) == kd.KD_ERR_INVALID_ARG
    # negative iterations / bad dtype / bad layout / ld too small
    assert kd.kd_decompose(1, 0, 0, 256, 4, 256, 0, -1, 0, 1, 1, 1, 1, null, null, null, null, null, 1, 1 << 20,
                           null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_decompose(1, 7, 0, 256, 4, 256, 0, 4, 0, 1, 1, 1, 1, null, null, null, null, null, 1, 1 << 20,
                           null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_decompose(1, 0, 5, 256, 4, 256, 0, 4, 0, 1, 1, 1, 1, null, null, null, null, null, 1, 1 << 20,
                           null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_decompose(1, 0, 0, 256, 4, 255, 0, 4, 0, 1, 1, 1, 1, null, null, null, null, null, 1, 1 << 20,
                           null) == kd.KD_ERR_INVALID_ARG
    # missing required outputs
    assert kd.kd_decompose(1, 0, 0, 256, 4, 256, 0, 4, 0, null, 1, 1, 1, null, null, null, null, null, 1, 1 << 20,
                           null) == kd.KD_ERR_INVALID_ARG
    # more blocks than the library accepts
    assert kd.kd_decompose(16, 0, 0, 256, 4, 256, 0, (1 << 16) + 1, 0, 16, 16, 16, 16, null, null, null, null, null,
                           16, 1 << 20, null) == kd.KD_ERR_INVALID_ARG
    # input or outputs not aligned to their elements
    assert kd.kd_decompose(2, 0, 0, 256, 4, 256, 0, 4, 0, 16, 16, 16, 16, null, null, null, null, null, 16, 1 << 20,
                           null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_decompose(16, 0, 0, 256, 4, 256, 0, 4, 0, 16, 18, 16, 16, null, null, null, null, null, 16, 1 << 20,
                           null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_decompose(16, 0, 0, 256, 4, 256, 0, 4, 0, 16, 16, 16, 16, null, 6, null, null, null, 16, 1 << 20,
                           null) == kd.KD_ERR_INVALID_ARG
    # workspace missing / too small
    assert kd.kd_decompose(16, 0, 0, 256, 4, 256, 0, 4, 0, 16, 16, 16, 16, null, null, null, null, null, null, 1 << 20,
                           null) == kd.KD_ERR_WORKSPACE
    assert kd.kd_decompose(16, 0, 0, 256, 4, 256, 0, 4, 0, 16, 16, 16, 16, null, null, null, null, null, 16, 16,
                           null) == kd.KD_ERR_WORKSPACE
    # workspace not 16-byte aligned (its tables are read with 128-bit loads)
    assert kd.kd_decompose(16, 0, 0, 256, 4, 256, 0, 4, 0, 16, 16, 16, 16, null, null, null, null, null, 8, 1 << 20,
                           null) == kd.KD_ERR_WORKSPACE
    assert kd.kd_apply_p(16, 16, 256, 2, 0, null, 0, null) == kd.KD_ERR_WORKSPACE
    assert kd.kd_apply_p(16, 6, 256, 2, 0, 16, 1 << 20, null) == kd.KD_ERR_INVALID_ARG   # y not 4-byte aligned
    assert kd.kd_apply_p(null, 1, 256, 2, 0, 1, 1 << 20, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_reconstruct(1, 1, 1, 1, 256, 2, 0, 9, 0, 1, 256, 1, 1 << 20, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_read_status(null, null) == kd.KD_ERR_WORKSPACE
    # batched reconstruct: matrix count and array
    assert kd.kd_reconstruct_batch(null, 1, 256, 0, 0, 16, 1 << 20, null) == kd.KD_ERR_INVALID_ARG
    recs = (kd.KdRecMat * 2)()
    assert kd.kd_reconstruct_batch(ctypes.cast(recs, ctypes.c_void_p), 0, 256, 0, 0, 16, 1 << 20,
                                   null) == kd.KD_ERR_INVALID_ARG
    recs[0] = kd.KdRecMat(16, 16, 16, 16, 0, 16, 4, 256)
    assert kd.kd_reconstruct_batch(ctypes.cast(recs, ctypes.c_void_p), 1, 4094, 0, 0, 16, 1 << 20,
                                   null) == kd.KD_ERR_UNSUPPORTED_N
    recs[0] = kd.KdRecMat(16, 16, 8, 16, 0, 16, 4, 256)   # centres not 16-byte aligned
    assert kd.kd_reconstruct_batch(ctypes.cast(recs, ctypes.c_void_p), 1, 256, 0, 0, 16, 1 << 20,
                                   null) == kd.KD_ERR_INVALID_ARG
    # batched dequantise: plane count and array
    assert kd.kd_dequantise_batch(null, 1, 256, 0, 0, null) == kd.KD_ERR_INVALID_ARG
    planes = (kd.KdPlane * 2)()
    assert kd.kd_dequantise_batch(ctypes.cast(planes, ctypes.c_void_p), 0, 256, 0, 0, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_dequantise_batch(ctypes.cast(planes, ctypes.c_void_p), kd.KD_MAX_BATCH + 1, 256, 0, 0,
                                  null) == kd.KD_ERR_INVALID_ARG
    # a plane with m > 0 and null pointers, then one whose ld is too small
    planes[0] = kd.KdPlane(None, None, None, 4, 256)
    assert kd.kd_dequantise_batch(ctypes.cast(planes, ctypes.c_void_p), 1, 256, 0, 0, null) == kd.KD_ERR_INVALID_ARG
    planes[0] = kd.KdPlane(16, 16, 16, 4, 255)
    assert kd.kd_dequantise_batch(ctypes.cast(planes, ctypes.c_void_p), 1, 256, 0, 0, null) == kd.KD_ERR_INVALID_ARG


def test_rht_block_and_validation(kd):
    for n in (16, 48, 768, 3072, 4096, 11008, 14336, 16384, 32768, 65536):
        assert kd.kd_rht_block(n) == ko.rht_block(n)
    for n in (0, 8, 24, 100, 65552, 131072):
        assert kd.kd_rht_block(n) == 0
    null = None
    assert kd.kd_rht(1, 0, 100, 4, 100, 0, 0, 1, 100, null, null) == kd.KD_ERR_UNSUPPORTED_N
    assert kd.kd_rht(1, 0, 256, -1, 256, 0, 0, 1, 256, null, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_rht(1, 0, 256, 4, 255, 0, 0, 1, 256, null, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_rht(1, 0, 256, 4, 256, 0, 0, 1, 255, null, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_rht(1, 9, 256, 4, 256, 0, 0, 1, 256, null, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_rht(1, 0, 256, 4, 256, 0, 2, 1, 256, null, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_rht(null, 0, 256, 4, 256, 0, 0, 1, 256, null, null) == kd.KD_ERR_INVALID_ARG
    # in place only for fp32 with equal strides
    assert kd.kd_rht(4096, 1, 256, 4, 256, 0, 0, 4096, 256, null, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_rht(4096, 0, 256, 4, 256, 0, 0, 4096, 512, null, null) == kd.KD_ERR_INVALID_ARG
    # pointers not aligned to their elements
    assert kd.kd_rht(4098, 0, 256, 4, 256, 0, 0, 8192, 256, null, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_rht(4097, 1, 256, 4, 256, 0, 0, 8192, 256, null, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_rht(4096, 1, 256, 4, 256, 0, 0, 8194, 256, null, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_rht(4096, 1, 256, 4, 256, 0, 0, 8192, 256, 6, null) == kd.KD_ERR_INVALID_ARG
    # nothing to do: no launch, no device needed
    assert kd.kd_rht(null, 0, 256, 0, 256, 0, 0, null, 256, null, null) == kd.KD_OK


def test_batch_workspace_and_validation(kd):
    import ctypes
    for n in (256, 768, 4096):
        one = kd.kd_workspace_size(n)
        assert kd.kd_workspace_size_batch(n, 1) == one
        big = kd.kd_workspace_size_batch(n, 32)
        assert big > one and big >= 256 + 32 * (n // 8) + 8 * n   # status, 32 sign sets, twiddles
    assert kd.kd_workspace_size_batch(4096, 0) == 0 and kd.kd_workspace_size_batch(4096, 33) == 0
    assert kd.kd_workspace_size_batch(4094, 2) == 0
    arr = (kd.KdMatrix * 2)()
    for i in range(2):
        arr[i] = kd.KdMatrix(None, 0, 4096, i, None, None, None, None, None)
    ptr = ctypes.cast(arr, ctypes.c_void_p)
    null = None
    assert kd.kd_decompose_batch(ptr, 0, 0, 0, 4096, 4, 0, 1, 1 << 30, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_decompose_batch(ptr, 33, 0, 0, 4096, 4, 0, 1, 1 << 30, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_decompose_batch(null, 2, 0, 0, 4096, 4, 0, 1, 1 << 30, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_decompose_batch(ptr, 2, 0, 0, 4094, 4, 0, 1, 1 << 30, null) == kd.KD_ERR_UNSUPPORTED_N
    assert kd.kd_decompose_batch(ptr, 2, 0, 0, 4096, 4, 0, 1, 16, null) == kd.KD_ERR_WORKSPACE
    arr[1] = kd.KdMatrix(None, 3, 4096, 1, None, None, None, None, None)   # m > 0 without pointers
    assert kd.kd_decompose_batch(ptr, 2, 0, 0, 4096, 4, 0, 1, 1 << 30, null) == kd.KD_ERR_INVALID_ARG
    arr[1] = kd.KdMatrix(1, 3, 4095, 1, 1, 1, 1, 1, None)                  # ld < n
    assert kd.kd_decompose_batch(ptr, 2, 0, 0, 4096, 4, 0, 1, 1 << 30, null) == kd.KD_ERR_INVALID_ARG


def test_dequantise_validation(kd):
    null = None
    assert kd.kd_dequantise(16, 16, 0, 4, 0, 0, 16, 16, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_dequantise(16, 16, 64, 4, 5, 0, 16, 64, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_dequantise(16, 16, 64, 4, 0, 3, 16, 64, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_dequantise(16, 16, 64, 4, 0, 0, 16, 63, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_dequantise(16, 16, 64, 4, 0, 1, 16, 3, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_dequantise(null, 16, 64, 4, 0, 0, 16, 64, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_dequantise(16, 8, 64, 4, 0, 0, 16, 64, null) == kd.KD_ERR_INVALID_ARG   # centres unaligned
    assert kd.kd_dequantise(null, null, 64, 0, 0, 0, null, 64, null) == kd.KD_OK


def test_product_path_requires_library(tmp_path, monkeypatch):
    """Importing the binding without the built library raises: no CPU fallback."""
    import importlib.util
    import shutil
    pkg = tmp_path / "pkgcopy"
    pkg.mkdir()
    src = os.path.join(ROOT, "paper_2609_11687_gb300", "kashin.py")
    shutil.copy(src, pkg / "kashin.py")
    spec = importlib.util.spec_from_file_location("kashin_nolib", pkg / "kashin.py")
    mod = importlib.util.module_from_spec(spec)
    with pytest.raises(ImportError):
        spec.loader.exec_module(mod)


def test_batch_wrappers_validate_counts_on_the_host(kd):
    """The batched wrappers refuse an empty batch, more than KD_MAX_BATCH entries and
    seed lists of the wrong length before they touch any device memory."""
    with pytest.raises(ValueError):
        kd.dequantise_batch([], 256)
    with pytest.raises(ValueError):
        kd.dequantise_batch([(None, None)] * (kd.KD_MAX_BATCH + 1), 256)
    with pytest.raises(ValueError):
        kd.reconstruct_batch([None, None], 256, [1])
    with pytest.raises(ValueError):
        kd.reconstruct_batch([None] * (kd.KD_MAX_BATCH + 1), 256, list(range(kd.KD_MAX_BATCH + 1)))
    with pytest.raises(ValueError):
        kd.decompose_batch([None, None], 4, [1])


def test_static_entry_checks_arguments_before_its_limit(kd):
    """kd_decompose_static checks the caller's arguments in kd_decompose's order and
    with its codes before applying its own length limit; none of these calls touches
    the GPU (the array's address is resolved only after every check passed)."""
    null = None
    st = kd.kd_decompose_static
    # a bad enum, a bad count or an unsupported length win over the length limit
    assert st(16, 7, 0, 16384, 4, 16384, 0, 4, 0, 16, 16, 16, 16, null, null, null, null, null,
              null) == kd.KD_ERR_INVALID_ARG
    assert st(16, 0, 0, 16384, 4, 16384, 0, -1, 0, 16, 16, 16, 16, null, null, null, null, null,
              null) == kd.KD_ERR_INVALID_ARG
    assert st(16, 0, 0, 16382, 4, 16382, 0, 4, 0, 16, 16, 16, 16, null, null, null, null, null,
              null) == kd.KD_ERR_UNSUPPORTED_N
    # ld too small, a null required output, an unaligned pointer
    assert st(16, 0, 0, 11008, 4, 100, 0, 4, 0, 16, 16, 16, 16, null, null, null, null, null,
              null) == kd.KD_ERR_INVALID_ARG
    assert st(16, 0, 0, 11008, 4, 11008, 0, 4, 0, 16, null, 16, 16, null, null, null, null, null,
              null) == kd.KD_ERR_INVALID_ARG
    assert st(16, 0, 0, 11008, 4, 11008, 0, 4, 0, 16, 16, 18, 16, null, null, null, null, null,
              null) == kd.KD_ERR_INVALID_ARG
    # valid arguments beyond the static array's limit
    assert st(16, 0, 0, 11008, 4, 11008, 0, 4, 0, 16, 16, 16, 16, null, null, null, null, null,
              null) == kd.KD_ERR_WORKSPACE


def test_host_entry_validates_before_copying(kd):
    """kd_decompose_batch_host refuses bad arguments and staging without a CUDA call."""
    null = None
    mats = (kd.KdMatrixHost * 2)()
    mats[0] = kd.KdMatrixHost(16, 4, 256, 0, 16, 16, 16, 16, None)
    mats[1] = kd.KdMatrixHost(16, 6, 256, 0, 16, 16, 16, 16, None)
    arr = ctypes.cast(mats, ctypes.c_void_p)
    f = kd.kd_decompose_batch_host
    assert kd.kd_staging_size_host(arr, 2, kd.KD_F16, kd.KD_VEC_ROWS, 256) > 0
    assert kd.kd_staging_size_host(arr, 0, kd.KD_F16, kd.KD_VEC_ROWS, 256) == 0
    assert f(null, 1, 1, 0, 256, 4, 0, 256, 1 << 30, 16, 1 << 20, null) == kd.KD_ERR_INVALID_ARG
    assert f(arr, 2, 9, 0, 256, 4, 0, 256, 1 << 30, 16, 1 << 20, null) == kd.KD_ERR_INVALID_ARG
    assert f(arr, 2, 1, 0, 4094, 4, 0, 256, 1 << 30, 16, 1 << 20, null) == kd.KD_ERR_UNSUPPORTED_N
    assert f(arr, 2, 1, 0, 256, -1, 0, 256, 1 << 30, 16, 1 << 20, null) == kd.KD_ERR_INVALID_ARG
    # staging null, unaligned or short; workspace short
    assert f(arr, 2, 1, 0, 256, 4, 0, null, 1 << 30, 16, 1 << 20, null) == kd.KD_ERR_WORKSPACE
    assert f(arr, 2, 1, 0, 256, 4, 0, 128, 1 << 30, 16, 1 << 20, null) == kd.KD_ERR_WORKSPACE
    assert f(arr, 2, 1, 0, 256, 4, 0, 256, 64, 16, 1 << 20, null) == kd.KD_ERR_WORKSPACE
    assert f(arr, 2, 1, 0, 256, 4, 0, 256, 1 << 30, 16, 8, null) == kd.KD_ERR_WORKSPACE
    # a matrix with m > 0 and a null output, then one whose ld is too small
    mats[1] = kd.KdMatrixHost(16, 6, 256, 0, None, 16, 16, 16, None)
    assert f(arr, 2, 1, 0, 256, 4, 0, 256, 1 << 30, 16, 1 << 20, null) == kd.KD_ERR_INVALID_ARG
    mats[1] = kd.KdMatrixHost(16, 6, 255, 0, 16, 16, 16, 16, None)
    assert f(arr, 2, 1, 0, 256, 4, 0, 256, 1 << 30, 16, 1 << 20, null) == kd.KD_ERR_INVALID_ARG


def test_matmul_2bit_validation(kd):
    """kd_matmul_2bit refuses bad sizes, null and unaligned pointers without a CUDA call."""
    f = kd.kd_matmul_2bit
    null = None
    assert f(16, 16, 16, 16, 0, 4, 16, 16, 1, 256, 16, 4, null) == kd.KD_ERR_INVALID_ARG       # n = 0
    assert f(16, 16, 16, 16, 256, 4, 16, 16, 1, 255, 16, 4, null) == kd.KD_ERR_INVALID_ARG     # ldx < n
    assert f(16, 16, 16, 16, 256, 4, 16, 16, 1, 256, 16, 3, null) == kd.KD_ERR_INVALID_ARG     # ldy < m
    assert f(16, 16, 16, 16, 256, 4, 16, 16, -1, 256, 16, 4, null) == kd.KD_ERR_INVALID_ARG    # batch < 0
    assert f(16, null, 16, 16, 256, 4, 16, 16, 1, 256, 16, 4, null) == kd.KD_ERR_INVALID_ARG
    assert f(16, 16, 8, 16, 256, 4, 16, 16, 1, 256, 16, 4, null) == kd.KD_ERR_INVALID_ARG      # centres 8-aligned
    assert f(16, 16, 16, 16, 256, 4, 18, 16, 1, 256, 16, 4, null) == kd.KD_ERR_INVALID_ARG     # x unaligned
    assert f(null, null, null, null, 256, 0, null, null, 1, 256, null, 0, null) == kd.KD_OK    # m == 0
    assert f(null, null, null, null, 256, 4, null, null, 0, 256, null, 4, null) == kd.KD_OK    # batch == 0


def test_matmul_2bit_f16_validation(kd):
    """kd_matmul_2bit_f16 refuses bad sizes, null and unaligned pointers (fp16 rows need
    2-byte alignment) without a CUDA call; its batched form refuses bad counts."""
    f = kd.kd_matmul_2bit_f16
    null = None
    assert f(16, 16, 16, 16, 0, 4, 16, 16, 1, 256, 16, 4, null) == kd.KD_ERR_INVALID_ARG       # n = 0
    assert f(16, 16, 16, 16, 256, 4, 16, 16, 1, 255, 16, 4, null) == kd.KD_ERR_INVALID_ARG     # ldx < n
    assert f(16, 16, 16, 16, 256, 4, 16, 16, 1, 256, 16, 3, null) == kd.KD_ERR_INVALID_ARG     # ldy < m
    assert f(16, 16, 16, 16, 256, 4, 16, 16, -1, 256, 16, 4, null) == kd.KD_ERR_INVALID_ARG    # batch < 0
    assert f(16, 16, 16, 16, 256, 4, 16, null, 1, 256, 16, 4, null) == kd.KD_ERR_INVALID_ARG   # xp null
    assert f(16, 16, 16, 8, 256, 4, 16, 16, 1, 256, 16, 4, null) == kd.KD_ERR_INVALID_ARG      # centres 8-aligned
    assert f(16, 16, 16, 16, 256, 4, 17, 16, 1, 256, 16, 4, null) == kd.KD_ERR_INVALID_ARG     # x odd address
    assert f(16, 16, 16, 16, 256, 4, 16, 16, 1, 256, 18, 4, null) == kd.KD_ERR_INVALID_ARG     # y unaligned
    assert f(null, null, null, null, 256, 0, null, null, 1, 256, null, 0, null) == kd.KD_OK    # m == 0
    assert f(null, null, null, null, 256, 4, null, null, 0, 256, null, 4, null) == kd.KD_OK    # batch == 0
    mats = (kd.KdFoldMatF16 * 2)()
    mats[0] = kd.KdFoldMatF16(16, 16, 16, 16, 16, 16, 16, 256, 4, 256, 4)
    mats[1] = kd.KdFoldMatF16(16, 16, 16, 16, 18, 16, 16, 256, 4, 255, 4)    # ldx < n
    arr = ctypes.cast(mats, ctypes.c_void_p)
    assert kd.kd_matmul_2bit_f16_batch(null, 1, 1, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_matmul_2bit_f16_batch(arr, 0, 1, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_matmul_2bit_f16_batch(arr, 33, 1, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_matmul_2bit_f16_batch(arr, 2, 1, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_matmul_2bit_f16_batch(arr, 2, 0, null) == kd.KD_ERR_INVALID_ARG       # checked even when empty
    assert kd.kd_matmul_2bit_f16_batch(arr, 1, 0, null) == kd.KD_OK
    fb = kd.kd_matmul_2bit_bf16
    assert fb(16, 16, 16, 16, 0, 4, 16, 16, 1, 256, 16, 4, null) == kd.KD_ERR_INVALID_ARG      # n = 0
    assert fb(16, 16, 16, 16, 256, 4, 17, 16, 1, 256, 16, 4, null) == kd.KD_ERR_INVALID_ARG    # x odd address
    assert fb(null, null, null, null, 256, 4, null, null, 0, 256, null, 4, null) == kd.KD_OK   # batch == 0
    assert kd.kd_matmul_2bit_bf16_batch(arr, 2, 1, null) == kd.KD_ERR_INVALID_ARG


def test_prepared_p_validation(kd):
    """kd_prepare_p and kd_apply_p_prepared refuse bad counts, null arrays, bad and
    unsupported lengths before any CUDA call."""
    null = None
    seeds = (ctypes.c_uint64 * 2)(1, 2)
    sp = ctypes.cast(seeds, ctypes.c_void_p)
    assert kd.kd_prepare_p(null, 1, 256, 16, 1 << 20, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_prepare_p(sp, 0, 256, 16, 1 << 20, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_prepare_p(sp, 33, 256, 16, 1 << 20, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_prepare_p(sp, 2, 0, 16, 1 << 20, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_prepare_p(sp, 2, 4094, 16, 1 << 20, null) == kd.KD_ERR_UNSUPPORTED_N
    pm = (kd.KdPMat * 2)()
    pm[0] = kd.KdPMat(16, 16, 4, 0)
    pm[1] = kd.KdPMat(16, 6, 4, 0)                                         # y not 4-byte aligned
    parr = ctypes.cast(pm, ctypes.c_void_p)
    assert kd.kd_apply_p_prepared(null, 1, 256, 16, 1 << 20, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_apply_p_prepared(parr, 0, 256, 16, 1 << 20, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_apply_p_prepared(parr, 1, 4094, 16, 1 << 20, null) == kd.KD_ERR_UNSUPPORTED_N
    assert kd.kd_apply_p_prepared(parr, 2, 256, 16, 1 << 20, null) == kd.KD_ERR_INVALID_ARG


def test_batched_product_and_transform_validation(kd):
    null = None
    mats = (kd.KdFoldMat * 2)()
    mats[0] = kd.KdFoldMat(16, 16, 16, 16, 16, 16, 16, 256, 4, 256, 4)
    mats[1] = kd.KdFoldMat(16, 16, 8, 16, 16, 16, 16, 256, 4, 256, 4)      # centres not 16-byte aligned
    arr = ctypes.cast(mats, ctypes.c_void_p)
    assert kd.kd_matmul_2bit_batch(null, 1, 1, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_matmul_2bit_batch(arr, 0, 1, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_matmul_2bit_batch(arr, 2, 1, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_matmul_2bit_batch(arr, 1, -1, null) == kd.KD_ERR_INVALID_ARG
    pm = (kd.KdPMat * 2)()
    pm[0] = kd.KdPMat(16, 16, 4, 1)
    pm[1] = kd.KdPMat(16, 6, 4, 2)                                         # y not 4-byte aligned
    parr = ctypes.cast(pm, ctypes.c_void_p)
    assert kd.kd_apply_p_batch(null, 1, 256, 16, 1 << 20, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_apply_p_batch(parr, 1, 4094, 16, 1 << 20, null) == kd.KD_ERR_UNSUPPORTED_N
    assert kd.kd_apply_p_batch(parr, 2, 256, 16, 1 << 20, null) == kd.KD_ERR_INVALID_ARG
    assert kd.kd_apply_p_batch(parr, 1, 256, null, 1 << 20, null) == kd.KD_ERR_WORKSPACE


def test_binding_leading_dimension_of_one_row(kd):
    """A one-row tensor may carry any row stride (numpy and torch treat it as contiguous
    either way); the binding then passes the row length as the leading dimension, which
    every entry point accepts.  Several rows keep their own stride."""
    import torch
    one = torch.zeros(10).as_strided((1, 10), (1, 1))
    assert kd._ld(one) == 10
    assert kd._ld(torch.zeros((3, 12))[:, :10]) == 12


def test_wrappers_refuse_bad_tensors_before_any_cuda_call(kd):
    """The tensor-level wrappers of the 16-bit product and of the prepared P check dtypes,
    shapes and counts on the host and raise ValueError before touching the device."""
    import pytest
    import torch

    class Planes:  # only the code-plane shape is read before the checks fail
        codes_u = torch.zeros((4, 16), dtype=torch.int32)

    d = [Planes()]
    f32, f16, bf16 = (torch.zeros((1, 256), dtype=t) for t in (torch.float32, torch.float16, torch.bfloat16))
    with pytest.raises(ValueError):
        kd.matmul_2bit_f16_batch(d, [f32], [f32])               # fp32 activations
    with pytest.raises(ValueError):
        kd.matmul_2bit_f16_batch(d, [f16], [bf16])              # mixed 16-bit types
    with pytest.raises(ValueError):
        kd.matmul_2bit_f16_batch(d, [torch.zeros((1, 240), dtype=torch.float16)] * 1,
                                 [torch.zeros((1, 240), dtype=torch.float16)])  # n does not match the planes
    with pytest.raises(ValueError):
        kd.prepare_p(256, list(range(33)))                      # more than 32 sign sets
    with pytest.raises(ValueError):
        kd.apply_p_prepared([f16], None)                        # P takes fp32 rows

